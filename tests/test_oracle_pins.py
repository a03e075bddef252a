"""Pins of the CPU oracle to facts outside itself (CPU only).

Each check ties an oracle function to the paper's definitions written out a
second, independent way (dense Kronecker matrices, an explicit damped inverse
solved by Cholesky, brute-force enumeration, closed forms, printed numbers).
The planted-mistake tests at the end show that plausible slips in the oracle
(a transposed factor, a wrong tie-break, a flipped zero sign, a dropped
damping normalisation, a wrong PCA order) make at least one pin fail.
"""
import math
import os

import numpy as np
import pytest
import scipy.linalg

from oracle import eogp_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def haar(d, rng):
    q, r = np.linalg.qr(rng.standard_normal((d, d)))
    return q * np.sign(np.diag(r))[None, :]


def vec(M):
    """Column-major vec."""
    return np.asarray(M).T.reshape(-1)


# ---------------------------------------------------------------- checks ---

def check_kronecker(Om, d_in, d_out, seed):
    """Q_A (x) Q_S as an explicit dense matrix: its transpose applied to vec(G)
    must equal the oracle's factored rotation, and it must diagonalise
    A (x) S with eigenvalues kron(lam_A, lam_S) (Sec. 2.2)."""
    rng = np.random.default_rng(seed)
    QA, QS = haar(d_in, rng), haar(d_out, rng)
    G = rng.standard_normal((d_out, d_in))
    K = np.kron(QA, QS)
    np.testing.assert_allclose(K.T @ vec(G), vec(Om.rotate(G, QA, QS)), atol=1e-12, rtol=0)
    lamA = np.sort(rng.uniform(0.1, 2.0, d_in))[::-1]
    lamS = np.sort(rng.uniform(0.1, 2.0, d_out))[::-1]
    A = QA @ np.diag(lamA) @ QA.T
    S = QS @ np.diag(lamS) @ QS.T
    ev = np.kron(lamA, lamS)
    np.testing.assert_allclose(np.kron(A, S) @ K, K * ev[None, :], atol=1e-12, rtol=0)
    Lam = Om.kfac_eigenvalues(lamS, lamA)
    np.testing.assert_array_equal(vec(Lam), ev)


def check_gradient_as_kron_sum(Om, seed):
    """vec(sum_t s_t a_t^T) = sum_t a_t (x) s_t, the per-token gradient whose
    second moment is E[(a a^T) (x) (delta delta^T)] (Eq. kfac_factorization)."""
    rng = np.random.default_rng(seed)
    T, d_in, d_out = 7, 5, 4
    a, s = rng.standard_normal((T, d_in)), rng.standard_normal((T, d_out))
    g = sum(np.kron(a[t], s[t]) for t in range(T))
    np.testing.assert_allclose(vec(Om.per_example_gradient(a, s)), g, atol=1e-12, rtol=0)


def check_selection(Om, lamA, lamS, m):
    """Brute force: stable descending order of the Kronecker eigenvalue vector,
    ties by Kronecker column position (pure-python sort on tuples)."""
    d_in, d_out = len(lamA), len(lamS)
    ev = [lamA[i] * lamS[j] for i in range(d_in) for j in range(d_out)]  # pos i*d_out+j
    order = sorted(range(len(ev)), key=lambda p: (-ev[p], p))[:m]
    j, i = Om.select_retained(Om.kfac_eigenvalues(lamS, lamA), m)
    assert list(i * d_out + j) == order


def check_first_stage_dense(Om, seed, d_in=6, d_out=5, m=11, T=9, B=3):
    """Eq. first_stage with Q_m built as explicit columns of Q_A (x) Q_S."""
    rng = np.random.default_rng(seed)
    QA, QS = haar(d_in, rng), haar(d_out, rng)
    Lam = rng.uniform(0.01, 3.0, (d_out, d_in))
    lam = 0.05
    a, s = rng.standard_normal((B, T, d_in)), rng.standard_normal((B, T, d_out))
    K = np.kron(QA, QS)
    ev = vec(Lam)
    order = sorted(range(d_in * d_out), key=lambda p: (-ev[p], p))[:m]
    Qm = K[:, order]
    z = Om.first_stage(a, s, QA, QS, Lam, lam, m)
    for b in range(B):
        g = vec(s[b].T @ a[b])
        zd = np.diag(1.0 / np.sqrt(ev[order] + lam)) @ Qm.T @ g
        np.testing.assert_allclose(z[b], zd, atol=1e-12, rtol=0)


def check_exact_influence(Om, seed, d_in, d_out, product_spectrum, P_kind):
    """Keep every coordinate and skip quantisation: <y, x> must equal the damped
    EK-FAC influence q^T (Q Lam Q^T + lam I)^{-1} g (Eq. practical_if with the
    EK-FAC curvature of Eq. ekfac_eigendecompose), solved here by Cholesky on
    the explicit d x d matrix."""
    rng = np.random.default_rng(seed)
    d = d_in * d_out
    QA, QS = haar(d_in, rng), haar(d_out, rng)
    if product_spectrum:
        Lam = Om.kfac_eigenvalues(np.sort(rng.uniform(0.01, 1, d_out))[::-1],
                                  np.sort(rng.uniform(0.01, 1, d_in))[::-1])
    else:
        Lam = rng.uniform(1e-3, 2.0, (d_out, d_in))
    lam = Om.damping(Lam, 0.1)
    P = np.eye(d) if P_kind == "identity" else haar(d, rng)
    T1, T2 = 6, 4
    a, s = rng.standard_normal((2, T1, d_in)), rng.standard_normal((2, T1, d_out))
    aq, sq = rng.standard_normal((1, T2, d_in)), rng.standard_normal((1, T2, d_out))
    x = Om.project(Om.first_stage(a, s, QA, QS, Lam, lam, d), P)
    y = Om.project(Om.first_stage(aq, sq, QA, QS, Lam, lam, d), P)
    got = Om.score_fp(x, y)[0]
    K = np.kron(QA, QS)
    H = K @ np.diag(vec(Lam)) @ K.T + lam * np.eye(d)
    cf = scipy.linalg.cho_factor(H)
    q = vec(sq[0].T @ aq[0])
    for b in range(2):
        g = vec(s[b].T @ a[b])
        want = q @ scipy.linalg.cho_solve(cf, g)
        assert abs(got[b] - want) <= 1e-10 * abs(want) + 1e-13


def check_damping(Om):
    """Eq. app_module_damping: lambda = 0.1 tr(Lam) / d."""
    Lam = np.full((3, 4), 2.0)
    assert Om.damping(Lam, 0.1) == pytest.approx(0.2, rel=1e-15)
    Lam = np.arange(1.0, 7.0).reshape(2, 3)   # trace 21, d = 6
    assert Om.damping(Lam, 0.1) == pytest.approx(0.35, rel=1e-15)


def check_pca_optimal(Om, seed, n=60, m=9, k=3):
    """Prop. 1 / App. A.1: the fitted top-k subspace attains the minimum
    reconstruction error sum_{j>k} mu_j, and beats random k-dim subspaces."""
    rng = np.random.default_rng(seed)
    Z = rng.standard_normal((n, m)) * (np.arange(1, m + 1) ** -0.8)[None, :]
    Z = Z @ haar(m, rng).T
    P, mu = Om.fit_pca(Z, k)
    C = Z.T @ Z / n
    allmu = np.sort(np.linalg.eigvalsh(C))[::-1]
    err = np.mean(np.sum((Z - Z @ P @ P.T) ** 2, axis=1))
    assert err == pytest.approx(allmu[k:].sum(), rel=1e-10)
    np.testing.assert_allclose(mu, allmu[:k], rtol=1e-10)
    for _ in range(50):
        W = np.linalg.qr(rng.standard_normal((m, k)))[0]
        assert np.mean(np.sum((Z - Z @ W @ W.T) ** 2, axis=1)) >= err - 1e-12


def check_eig_closed_forms(Om):
    """Closed-form spectra: a diagonal second moment and a rotated 2x2 one."""
    dvals = np.array([0.5, 3.0, 1.0, 2.0])
    Z = np.diag(np.sqrt(4 * dvals))           # n = m = 4: Z^T Z / n = diag(dvals)
    P, mu = Om.fit_pca(Z, 3, route="cov")
    np.testing.assert_allclose(mu, [3.0, 2.0, 1.0], rtol=1e-12)
    np.testing.assert_allclose(np.abs(P), np.eye(4)[:, [1, 3, 2]], atol=1e-12)
    assert np.all(P[[1, 3, 2], [0, 1, 2]] > 0)      # canonical sign: largest entry positive
    th = 0.3
    R = np.array([[math.cos(th), -math.sin(th)], [math.sin(th), math.cos(th)]])
    C = R @ np.diag([3.0, 1.0]) @ R.T
    Z = np.linalg.cholesky(2 * C).T            # Z^T Z / 2 = C
    P, mu = Om.fit_pca(Z, 1, route="cov")
    assert mu[0] == pytest.approx(3.0, rel=1e-12)
    np.testing.assert_allclose(P[:, 0], R[:, 0] * np.sign(R[np.argmax(np.abs(R[:, 0])), 0]),
                               atol=1e-12)


def check_gram_route(Om, seed):
    """App. B.2: directions from the n x n Gram matrix equal those from Z^T Z / n."""
    rng = np.random.default_rng(seed)
    Z = rng.standard_normal((20, 50)) * (np.arange(1, 51) ** -0.5)[None, :]
    P1, mu1 = Om.fit_pca(Z, 6, route="gram")
    P2, mu2 = Om.fit_pca(Z, 6, route="cov")
    np.testing.assert_allclose(mu1, mu2, rtol=1e-10)
    np.testing.assert_allclose(P1, P2, atol=1e-9)


def check_prop2(Om, seed, d_in=6, d_out=5, m=12, k=4, n=80):
    """Prop. 2 / App. A.2: PCA within span(Q_m) reconstructs the full-space
    half-whitened gradients no worse than the leading k EK-FAC axes, and the
    error splits as in Eq. app_restricted_reconstruction."""
    rng = np.random.default_rng(seed)
    QA, QS = haar(d_in, rng), haar(d_out, rng)
    Lam = rng.uniform(0.05, 2.0, (d_out, d_in))
    lam = Om.damping(Lam, 0.1)
    a = rng.standard_normal((n, 3, d_in)) * rng.uniform(0.2, 2, d_in)[None, None, :]
    s = rng.standard_normal((n, 3, d_out))
    K = np.kron(QA, QS)
    ev = vec(Lam)
    Hm12 = K @ np.diag(1 / np.sqrt(ev + lam)) @ K.T      # Eq. ekfac_half_whitening
    X = np.stack([Hm12 @ vec(s[b].T @ a[b]) for b in range(n)])
    z = Om.first_stage(a, s, QA, QS, Lam, lam, m)
    order = sorted(range(d_in * d_out), key=lambda p: (-ev[p], p))[:m]
    Qm = K[:, order]
    np.testing.assert_allclose(z, X @ Qm, atol=1e-10)    # a_i = Q_m^T x_i
    P, _ = Om.fit_pca(z, k)
    U = Qm @ P
    Qk = Qm[:, :k]
    e_pca = np.mean(np.sum((X - X @ U @ U.T) ** 2, axis=1))
    e_ek = np.mean(np.sum((X - X @ Qk @ Qk.T) ** 2, axis=1))
    assert e_pca <= e_ek + 1e-12
    e_out = np.mean(np.sum((X - X @ Qm @ Qm.T) ** 2, axis=1))
    e_in = np.mean(np.sum((z - z @ P @ P.T) ** 2, axis=1))
    assert e_pca == pytest.approx(e_out + e_in, rel=1e-10)


def check_onebit(Om, seed):
    """Eq. onebit and App. A.3: s = ||x||_1/k minimises ||x - s b||^2, and the
    closed form of Eq. app_onebit_scale holds; zeros of either sign map to +1."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((1, 37))
    bits, s = Om.onebit(x)
    b = np.where(bits[0], 1.0, -1.0)
    np.testing.assert_array_equal(b, np.sign(x[0]))
    k = x.shape[1]
    l1, l2 = np.abs(x).sum(), (x ** 2).sum()
    for t in np.linspace(0, 2 * s[0], 41):
        e = ((x[0] - t * b) ** 2).sum()
        assert e >= ((x[0] - s[0] * b) ** 2).sum() - 1e-12
        assert e == pytest.approx(k * (t - l1 / k) ** 2 + l2 - l1 ** 2 / k, rel=1e-12, abs=1e-12)
    bz, _ = Om.onebit(np.array([[0.0, -0.0, 1e-300, -1e-300, 5.0, -5.0]]))
    assert bz[0].tolist() == [True, True, True, False, True, False]


def check_packing(Om, seed):
    """Round trip, zero pad bits, the paper's per-module byte order, and the
    popcount identity <b, b'> = k - 2 popc(b xor b') against explicit +-1 sums."""
    rng = np.random.default_rng(seed)
    for k in (1, 5, 31, 32, 33, 64, 100, 128, 1000):
        bits = rng.integers(0, 2, (4, k)).astype(bool)
        w = Om.pack_bits(bits)
        assert w.shape == (4, (k + 31) // 32) and w.dtype == np.uint32
        np.testing.assert_array_equal(Om.unpack_bits(w, k), bits)
        if k % 32:
            assert np.all((w[:, -1].astype(np.uint64) >> np.uint64(k % 32)) == 0)
        by = w.astype("<u4").view(np.uint8).reshape(4, -1)
        for c in range(k):
            assert np.all(((by[:, c // 8] >> (c % 8)) & 1) == bits[:, c])
        pm = np.where(bits, 1, -1)
        for r in range(3):
            h = sum(bin(int(x) ^ int(y)).count("1") for x, y in zip(w[r], w[r + 1]))
            assert int(pm[r] @ pm[r + 1]) == k - 2 * h


def check_scores(Om, seed):
    """Codes score: f32 order agrees with float64 within its bound; a paper-mode
    query equal to its own dequantised code reproduces the codes score; the
    codes score equals the popcount form."""
    rng = np.random.default_rng(seed)
    ks = [40, 64, 7]
    W = sum((k + 31) // 32 for k in ks)
    N, Q = 9, 4
    def rand_codes(n):
        return Om.pack_concat([rng.integers(0, 2, (n, k)).astype(bool) for k in ks])
    tc, qc = rand_codes(N), rand_codes(Q)
    ts = rng.lognormal(0, 0.5, (N, 3)).astype(np.float32)
    qs = rng.lognormal(0, 0.5, (Q, 3)).astype(np.float32)
    s64 = Om.score_codes(tc, ts, ks, qc, qs)
    s32 = Om.score_codes_f32(tc, ts, ks, qc, qs)
    bound = 1e-6 * sum(np.abs(qs[:, u, None] * ts[None, :, u]) * k for u, k in enumerate(ks))
    assert np.all(np.abs(s64 - s32) <= bound)
    off = Om.module_word_offsets(ks)
    for q in range(Q):
        for i in range(N):
            tot = 0.0
            for u, k in enumerate(ks):
                h = sum(bin(int(a) ^ int(b)).count("1")
                        for a, b in zip(tc[i, off[u]:off[u + 1]], qc[q, off[u]:off[u + 1]]))
                tot += float(qs[q, u]) * float(ts[i, u]) * (k - 2 * h)
            assert s64[q, i] == pytest.approx(tot, rel=1e-12, abs=1e-12)
    y = np.concatenate([np.where(Om.unpack_bits(qc[:, off[u]:off[u + 1]], k), 1.0, -1.0)
                        * qs[:, u, None] for u, k in enumerate(ks)], axis=1)
    np.testing.assert_allclose(Om.score_paper(tc, ts, ks, y), s64, rtol=1e-12, atol=1e-12)


# -------------------------------------------------------------- the tests ---

@pytest.mark.parametrize("d_in,d_out", [(8, 8), (12, 10), (16, 24)])
def test_kronecker_bruteforce(d_in, d_out):
    check_kronecker(O, d_in, d_out, seed=d_in * 100 + d_out)


def test_gradient_is_kron_sum():
    check_gradient_as_kron_sum(O, 3)


@pytest.mark.parametrize("m", [1, 6, 7, 10, 33, 64])
def test_selection_bruteforce_with_ties(m):
    lam = np.arange(1, 9, dtype=np.float64) ** -1.5     # symmetric product: exact ties
    check_selection(O, lam, lam, m)
    check_selection(O, np.arange(1, 7.0) ** -1.0, np.arange(1, 5.0) ** -1.0, min(m, 24))


def test_first_stage_dense_definition():
    check_first_stage_dense(O, 7)


@pytest.mark.parametrize("d_in,d_out,product,P_kind", [
    (6, 5, True, "identity"), (6, 5, False, "orthogonal"), (8, 8, True, "orthogonal"),
    (8, 8, False, "identity")])
def test_full_keep_equals_exact_ekfac_influence(d_in, d_out, product, P_kind):
    check_exact_influence(O, 11 + d_in, d_in, d_out, product, P_kind)


def test_damping_rule():
    check_damping(O)


def test_prop1_pca_optimal_value():
    check_pca_optimal(O, 5)


def test_eigensolver_closed_forms():
    check_eig_closed_forms(O)


def test_gram_route_equals_covariance_route():
    check_gram_route(O, 9)


def test_prop2_eigenbasis_correction():
    check_prop2(O, 13)


def test_onebit_scale_and_zero_sign():
    check_onebit(O, 17)


def test_packing_and_popcount_identity():
    check_packing(O, 19)


def test_scores():
    check_scores(O, 23)


@pytest.mark.parametrize("counter", ["bitwise_count", "byte_table"])
def test_onebit_dot_xor_equals_pm1_sums(counter, monkeypatch):
    """The XOR / population-count form of the one-bit inner product equals the
    explicit +-1 sum, for ragged and word-multiple k (both counting routes)."""
    if counter == "byte_table":
        monkeypatch.delattr(np, "bitwise_count", raising=False)
    rng = np.random.default_rng(41)
    for k in (1, 31, 32, 33, 100, 1024, 2049):
        bt = rng.integers(0, 2, (50, k)).astype(bool)
        bq = rng.integers(0, 2, (3, k)).astype(bool)
        tw, qw = O.pack_bits(bt), O.pack_bits(bq)
        for q in range(3):
            want = np.where(bt, 1, -1) @ np.where(bq[q], 1, -1)
            np.testing.assert_array_equal(O.onebit_dot_xor(tw, qw[q], k), want)


def test_norm_preservation():
    """An orthogonal rotation preserves the Frobenius norm and inner products."""
    rng = np.random.default_rng(29)
    QA, QS = haar(12, rng), haar(9, rng)
    G1, G2 = rng.standard_normal((9, 12)), rng.standard_normal((9, 12))
    R1, R2 = O.rotate(G1, QA, QS), O.rotate(G2, QA, QS)
    assert np.linalg.norm(R1) == pytest.approx(np.linalg.norm(G1), rel=1e-12)
    assert np.sum(R1 * R2) == pytest.approx(np.sum(G1 * G2), rel=1e-12)


def check_topk(Om, seed):
    """Ranking by brute force: Python's sort of (-score, index) pairs over the
    non-NaN scores, on rows with planted ties, NaNs, -inf and fewer rows than K."""
    rng = np.random.default_rng(seed)
    Q, N, K = 6, 23, 8
    sc = rng.integers(-4, 5, (Q, N)).astype(np.float64)   # many equal scores
    sc[1, ::3] = np.nan
    sc[2, :] = np.nan
    sc[2, 5] = 1.5
    sc[3, 7] = -np.inf
    sc[4] = rng.standard_normal(N)
    for Kq, rows in ((K, sc), (30, sc[:2])):               # K > N: tail must be (-inf, -1)
        vals, idx = Om.top_k(rows, Kq)
        for q in range(rows.shape[0]):
            pairs = sorted((-rows[q, i], i) for i in range(rows.shape[1]) if not math.isnan(rows[q, i]))
            want = pairs[:Kq]
            assert [int(i) for i in idx[q, :len(want)]] == [i for _, i in want]
            assert list(vals[q, :len(want)]) == [-v for v, _ in want]
            assert (idx[q, len(want):] == -1).all() and (vals[q, len(want):] == -np.inf).all()


def test_topk_brute_force():
    check_topk(O, 31)


def check_srht(Om, seed):
    """SRHT pins: the Hadamard entries against (-1)^popcount(r & c) by brute
    force; k = p with unit signs is the orthonormal H, so applying it twice is
    the identity and norms are kept; the sqrt(p/k) normalisation makes
    E ||S z||^2 = ||z||^2 over random row subsets (exact average over all
    subsets of size 1 for a tiny p); zero padding ignores the padded signs."""
    rng = np.random.default_rng(seed)
    for m in (1, 5, 8, 13):
        p = Om.srht_width(m)
        assert p >= m and p & (p - 1) == 0 and (p == 1 or p // 2 < m)
    p = 8
    z = rng.standard_normal((3, p))
    x = Om.srht(z, np.ones(p), np.arange(p))
    H = np.array([[(-1) ** bin(r & c).count("1") for c in range(p)] for r in range(p)]) / math.sqrt(p)
    np.testing.assert_allclose(x, z @ H.T, atol=1e-14, rtol=0)
    np.testing.assert_allclose(Om.srht(x, np.ones(p), np.arange(p)), z, atol=1e-13, rtol=0)
    np.testing.assert_allclose(np.linalg.norm(x, axis=1), np.linalg.norm(z, axis=1), rtol=1e-13)
    # average of ||S z||^2 over every single-row selection equals ||z||^2
    sg = rng.choice([-1.0, 1.0], p)
    avg = np.mean([np.sum(Om.srht(z, sg, [r]) ** 2, axis=1) for r in range(p)], axis=0)
    np.testing.assert_allclose(avg, np.sum(z ** 2, axis=1), rtol=1e-12)
    # m = 6 pads to p = 8; the signs are applied before padding, rows keep their order
    z6 = rng.standard_normal((2, 6))
    sg6 = rng.choice([-1.0, 1.0], 6)
    rows = np.array([5, 0, 3])
    want = math.sqrt(8 / 3) * (np.concatenate([z6 * sg6, np.zeros((2, 2))], 1) @ H.T)[:, rows]
    np.testing.assert_allclose(Om.srht(z6, sg6, rows), want, atol=1e-13, rtol=0)


def test_srht():
    check_srht(O, 37)


def check_ekfac(Om, seed):
    """EK-FAC correction pins: the squared coordinates of vec(G_b) under the
    dense Kronecker basis (Q_A (x) Q_S)^T, summed over examples; their total
    equals sum_b ||G_b||_F^2 (the basis is orthonormal); one token of one
    example gives the outer product of the squared rotated factors."""
    rng = np.random.default_rng(seed)
    B, T, d_in, d_out = 3, 4, 5, 6
    QA, QS = haar(d_in, rng), haar(d_out, rng)
    a, s = rng.standard_normal((B, T, d_in)), rng.standard_normal((B, T, d_out))
    got = Om.ekfac_sumsq(a, s, QA, QS)
    K = np.kron(QA, QS)
    want = sum((K.T @ vec(sum(np.outer(s[b, t], a[b, t]) for t in range(T)))) ** 2 for b in range(B))
    np.testing.assert_allclose(vec(got), want, rtol=1e-12, atol=1e-14)
    tot = sum(np.sum(sum(np.outer(s[b, t], a[b, t]) for t in range(T)) ** 2) for b in range(B))
    assert got.sum() == pytest.approx(tot, rel=1e-12)
    one = Om.ekfac_sumsq(a[:1, :1], s[:1, :1], QA, QS)
    np.testing.assert_allclose(one, np.outer((QS.T @ s[0, 0]) ** 2, (QA.T @ a[0, 0]) ** 2),
                               rtol=1e-12, atol=1e-15)


def test_ekfac_correction():
    check_ekfac(O, 41)


def check_plumbing(Om, seed):
    """Bias channel: the last column of G for [a; 1] is sum_t s_t and the other
    columns are G for a. Token lengths: G_b from the masked s equals the sum
    over the example's own tokens only."""
    rng = np.random.default_rng(seed)
    T, d_in, d_out = 6, 4, 3
    a, s = rng.standard_normal((2, T, d_in)), rng.standard_normal((2, T, d_out))
    ab = Om.with_bias_channel(a)
    assert ab.shape == (2, T, d_in + 1) and (ab[..., -1] == 1).all() and (ab[..., :-1] == a).all()
    G = Om.per_example_gradient(ab[0], s[0])
    np.testing.assert_allclose(G[:, -1], s[0].sum(0), rtol=1e-13)
    np.testing.assert_allclose(G[:, :-1], Om.per_example_gradient(a[0], s[0]), rtol=1e-13)
    sm = Om.mask_tokens(s, [4, 0])
    want = sum(np.outer(s[0, t], a[0, t]) for t in range(4))
    np.testing.assert_allclose(Om.per_example_gradient(a[0], sm[0]), want, rtol=1e-13)
    assert not Om.per_example_gradient(a[1], sm[1]).any()


def test_bias_channel_and_token_lengths():
    check_plumbing(O, 43)


def check_sharded_fit(Om, seed):
    """Summing the shards' second moments and fitting from the sum equals the
    fit on all rows (covariance route), with either shard order."""
    rng = np.random.default_rng(seed)
    Z = rng.standard_normal((50, 12)) * np.linspace(3, 0.2, 12)[None, :]
    parts = [Z[:17], Z[17:31], Z[31:]]
    C = sum(p.T @ p for p in parts)
    P, mu = Om.fit_pca_from_moment(C, 50, 5)
    P0, mu0 = Om.fit_pca(Z, 5, route="cov")
    np.testing.assert_allclose(mu, mu0, rtol=1e-12)
    np.testing.assert_allclose(P, P0, atol=1e-10)
    P2, _ = Om.fit_pca_from_moment(sum(p.T @ p for p in parts[::-1]), 50, 5)
    np.testing.assert_allclose(P2, P0, atol=1e-10)


def test_sharded_pca_fit():
    check_sharded_fit(O, 53)


def _golden_rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def test_payload_matches_tab_cost():
    for model, layers, per, k, kb in _golden_rows("tab_cost_payload.txt"):
        ks = [int(k)] * (int(layers) * int(per))
        assert O.payload_bytes(ks) == round(float(kb) * 1000), model
    assert O.payload_bytes([2048]) == 258


def check_payload(Om, seed):
    """Store records: the size of Eq. app_payload (pinned to Tab. cost above), the
    byte order of the signs written out by hand, the half-precision scale
    (round to nearest even) and the round trip."""
    rng = np.random.default_rng(seed)
    ks = [13, 32, 70]
    bits = [rng.integers(0, 2, (4, k)).astype(bool) for k in ks]
    codes = Om.pack_concat(bits)
    scales = np.array([[1.0, 1 + 2 ** -11, 1 + 3 * 2 ** -11]] * 4, np.float32)
    pay = Om.to_payload(codes, scales, ks)
    assert pay.shape == (4, Om.payload_bytes(ks))
    o = 0
    for u, k in enumerate(ks):
        nb = (k + 7) // 8
        for e in range(4):
            for c in range(k):
                assert ((int(pay[e, o + c // 8]) >> (c % 8)) & 1) == int(bits[u][e, c])
            assert int(pay[e, o + (k - 1) // 8]) >> ((k - 1) % 8 + 1) == 0   # pad bits are 0
        halfbits = int(pay[0, o + nb]) | (int(pay[0, o + nb + 1]) << 8)
        want = {0: 0x3C00, 1: 0x3C00, 2: 0x3C02}[u]   # 1, tie to even -> 1, 1 + 2^-9
        assert halfbits == want
        o += nb + 2
    c2, s2 = Om.from_payload(pay, ks)
    np.testing.assert_array_equal(c2, codes)
    np.testing.assert_array_equal(s2, scales.astype(np.float16).astype(np.float32))


def test_payload_records():
    check_payload(O, 47)


def test_correction_storage_matches_paper():
    for m, k, mods, gb, tol in _golden_rows("correction_storage.txt"):
        tot = O.correction_bytes(int(m), int(k)) * int(mods) / 1e9
        assert abs(tot - float(gb)) <= float(tol) * float(gb)


# ------------------------------------------------------ planted mistakes ---

def _fails(fn, *args, **kw):
    try:
        fn(*args, **kw)
    except (AssertionError, ValueError, IndexError):
        return True
    return False


def test_planted_transposed_rotation_is_caught(monkeypatch):
    # Q_A applied transposed (rows instead of columns as eigenvectors)
    monkeypatch.setattr(O, "rotate", lambda G, QA, QS: np.asarray(QS).T @ G @ np.asarray(QA).T)
    assert _fails(check_kronecker, O, 8, 8, 1)
    assert _fails(check_first_stage_dense, O, 7)


def test_planted_wrong_tiebreak_is_caught(monkeypatch):
    def bad(Lam, m):
        d_out, d_in = Lam.shape
        vals = Lam.reshape(-1)                 # row-major position j*d_in + i
        order = np.lexsort((np.arange(vals.size), -vals))[:m]
        return order // d_in, order % d_in
    monkeypatch.setattr(O, "select_retained", bad)
    lam = np.arange(1, 9, dtype=np.float64) ** -1.5
    assert _fails(check_selection, O, lam, lam, 7)


def test_planted_zero_sign_is_caught(monkeypatch):
    def bad(x):
        x = np.asarray(x, np.float64)
        return x > 0, np.abs(x).sum(axis=-1) / x.shape[-1]
    monkeypatch.setattr(O, "onebit", bad)
    assert _fails(check_onebit, O, 17)


def test_planted_damping_mistake_is_caught(monkeypatch):
    monkeypatch.setattr(O, "damping", lambda Lam, rel: float(rel * np.asarray(Lam).sum()))
    assert _fails(check_damping, O)


def test_planted_missing_scale_is_caught(monkeypatch):
    orig = O.first_stage
    def bad(a, s, QA, QS, Lam, lam, m):   # drops the (Lam + lam)^{-1/2} factor
        j, i = O.select_retained(Lam, m)
        return orig(a, s, QA, QS, Lam, lam, m) * np.sqrt(np.asarray(Lam)[j, i] + lam)[None, :]
    monkeypatch.setattr(O, "first_stage", bad)
    assert _fails(check_exact_influence, O, 3, 6, 5, True, "identity")


def test_planted_pca_order_is_caught(monkeypatch):
    orig = O.fit_pca
    def bad(Z, k, route="auto"):             # smallest instead of largest eigenvalues
        P, mu = orig(Z, Z.shape[1] if Z.shape[0] >= Z.shape[1] else Z.shape[0], route)
        return P[:, -k:], mu[-k:]
    monkeypatch.setattr(O, "fit_pca", bad)
    assert _fails(check_pca_optimal, O, 5)


def test_planted_bit_order_is_caught(monkeypatch):
    orig = O.pack_bits
    monkeypatch.setattr(O, "pack_bits", lambda b: orig(np.asarray(b)[..., ::-1]))
    assert _fails(check_packing, O, 19)


def test_planted_topk_mistakes_are_caught(monkeypatch):
    orig = O.top_k
    def later_index_first(scores, K):        # equal scores ranked by higher index
        v, i = orig(np.asarray(scores)[:, ::-1], K)
        n = np.asarray(scores).shape[1]
        return v, np.where(i >= 0, n - 1 - i, -1)
    monkeypatch.setattr(O, "top_k", later_index_first)
    assert _fails(check_topk, O, 31)

    def nan_ranks(scores, K):                # NaN treated as the lowest score instead of dropped
        return orig(np.nan_to_num(np.asarray(scores, np.float64), nan=-1e300), K)
    monkeypatch.setattr(O, "top_k", nan_ranks)
    assert _fails(check_topk, O, 31)


def test_planted_srht_mistakes_are_caught(monkeypatch):
    orig = O.srht
    monkeypatch.setattr(O, "srht", lambda z, sg, rows: orig(z, sg, rows) * math.sqrt(len(rows) / O.srht_width(np.asarray(z).shape[1])))
    assert _fails(check_srht, O, 37)          # normalisation dropped
    monkeypatch.setattr(O, "srht", lambda z, sg, rows: orig(z, -np.asarray(sg, np.float64), rows)[:, ::-1])
    assert _fails(check_srht, O, 37)          # rows reversed


def test_planted_ekfac_mistakes_are_caught(monkeypatch):
    orig = O.ekfac_sumsq
    monkeypatch.setattr(O, "ekfac_sumsq", lambda a, s, QA, QS: orig(a, s, QA, QS) / np.asarray(a).shape[0])
    assert _fails(check_ekfac, O, 41)         # mean instead of sum
    monkeypatch.setattr(O, "ekfac_sumsq", lambda a, s, QA, QS: orig(np.asarray(a)[:, ::-1], s, QA, QS))
    assert _fails(check_ekfac, O, 41)         # tokens of a and s paired wrongly


def test_planted_plumbing_mistakes_are_caught(monkeypatch):
    orig = O.mask_tokens
    monkeypatch.setattr(O, "mask_tokens", lambda s, n: orig(s, [int(x) + 1 for x in n]))
    assert _fails(check_plumbing, O, 43)      # off-by-one length
    monkeypatch.setattr(O, "mask_tokens", orig)
    ob = O.with_bias_channel
    monkeypatch.setattr(O, "with_bias_channel", lambda a: ob(a)[..., ::-1])
    assert _fails(check_plumbing, O, 43)      # bias channel first instead of last


def test_planted_payload_mistake_is_caught(monkeypatch):
    orig = O.to_payload
    def big_endian_half(codes, scales, ks):
        pay = orig(codes, scales, ks).copy()
        o = 0
        for k in ks:
            nb = (k + 7) // 8
            pay[:, [o + nb, o + nb + 1]] = pay[:, [o + nb + 1, o + nb]]
            o += nb + 2
        return pay
    monkeypatch.setattr(O, "to_payload", big_endian_half)
    assert _fails(check_payload, O, 47)


def test_planted_sharded_fit_mistake_is_caught(monkeypatch):
    orig = O.fit_pca_from_moment
    monkeypatch.setattr(O, "fit_pca_from_moment", lambda C, n, k: orig(C, 1, k))   # sum, not mean
    assert _fails(check_sharded_fit, O, 53)
