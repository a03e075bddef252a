"""GPU parity: every ABI call against the CPU oracle on identical seeded inputs.

Tolerances (the parity rules, written out here):
  * pre-sign coordinates z and x: per row ||x_gpu - x_oracle|| / ||x_oracle||
    <= 1e-5 for fp32 inputs, <= 2e-3 for bf16 inputs;
  * sign bits: bit-exact except coordinates with |x_oracle| < 1e-4 ||x_oracle||
    (the count is printed);
  * CODES scores: bit-exact against the oracle's fixed fp32 evaluation order;
  * scales ||x||_1/k: relative 1e-5 (fp32 accumulation of k terms).
"""
import numpy as np
import pytest

from oracle import eogp_oracle as O
from paper_2609_37842_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2609_37842_gb300 import eogp as E  # noqa: E402

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_37842_gb300 import build
    build.build()
    E.lib()
    yield
    E.sync_status()


def to_dev(x, dtype):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(DEV).to(dtype)


def codes_np(t):
    return t.cpu().numpy().view(np.uint32)


def row_rel(got, want):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    return np.linalg.norm(got - want, axis=1) / np.maximum(np.linalg.norm(want, axis=1), 1e-300)


def check_bits(x_or, codes, k):
    bits, _ = O.onebit(x_or)
    got = O.unpack_bits(codes, k)
    small = np.abs(x_or) < 1e-4 * np.linalg.norm(x_or, axis=1, keepdims=True)
    bad = (got != bits) & ~small
    assert not bad.any(), f"{bad.sum()} sign bits differ outside the exclusion band"
    flips = int(((got != bits) & small).sum())
    print(f"[signs] excluded coordinates: {int(small.sum())}, of which differing: {flips}")
    return flips


# ---------------------------------------------------------------- pack_sign

@pytest.mark.parametrize("B,k", [(1, 1), (7, 31), (5, 32), (300, 100), (64, 128), (33, 1000),
                                 (16, 1024), (3, 16384 + 96), (5000, 1024), (4100, 100)])
def test_pack_sign(B, k):
    rng = np.random.default_rng(B * 1000 + k)
    x = rng.standard_normal((B, k)).astype(np.float32)
    x[:, ::7] = 0.0
    x[:, 3::11] = -0.0
    xd = torch.from_numpy(x).to(DEV)
    W = (k + 31) // 32
    codes = torch.full((B, W + 3), -1, dtype=torch.int32, device=DEV)   # strided store rows
    scales = torch.full((B, 2), -1.0, dtype=torch.float32, device=DEV)
    E.pack_sign(xd, codes=codes[:, 1:W + 1], scales=scales[:, 1])
    E.sync_status()
    c = codes_np(codes)
    bits, sc = O.onebit(x.astype(np.float64))
    np.testing.assert_array_equal(c[:, 1:W + 1], O.pack_bits(bits))
    assert np.all(c[:, 0] == 0xFFFFFFFF) and np.all(c[:, W + 1:] == 0xFFFFFFFF)
    np.testing.assert_allclose(scales[:, 1].cpu().numpy(), sc, rtol=1e-5)
    assert np.all(scales[:, 0].cpu().numpy() == -1.0)
    # bitwise reproducible
    c2, s2 = E.pack_sign(xd)
    c3, s3 = E.pack_sign(xd)
    assert torch.equal(c2, c3) and torch.equal(s2, s3)


def test_pack_sign_nan_sets_device_status():
    x = torch.zeros((2, 64), device=DEV)
    x[1, 5] = float("nan")
    E.pack_sign(x)
    with pytest.raises(E.EOGPError) as ei:
        E.sync_status()
    assert ei.value.code == E.EDEVICE
    E.sync_status()  # cleared


# -------------------------------------------------------------------- score

def rand_store(rng, n, ks):
    return O.pack_concat([rng.integers(0, 2, (n, k)).astype(bool) for k in ks])


@pytest.mark.parametrize("N,Q,ks", [(1, 1, [32]), (300, 1, [40, 64, 7]), (257, 3, [1024]),
                                    (1000, 1, [128, 1024]), (513, 5, [256, 2048]),
                                    (1000, 8, [128, 5, 300]), (130, 9, [64, 64]),
                                    (513, 70, [40, 1024, 7, 33]), (64, 64, [16384]),
                                    (1000, 64, [128, 1024]), (300, 100, [256]),
                                    (129, 200, [1024, 128, 2048]), (777, 257, [512] * 5),
                                    (1000, 300, [256, 768, 1024]), (500, 300, [2048]),
                                    (2000, 64, [256, 1280]), (5000, 200, [768]), (40000, 64, [1024]),
                                    (70000, 64, [4096]), (3000, 64, [768]),
                                    (3000, 1000, [256, 256, 512])])
@pytest.mark.parametrize("f4", ["1", "0"])
def test_score_codes_bit_exact(N, Q, ks, f4, eogp_options):
    """CODES scores equal the oracle's float32 evaluation bit for bit. Where every
    module is a multiple of 256 bits the tensor-core kernel takes e2m1 operands
    (kind::mxf4, unit scales) unless EOGP_OPT_SCORE_OPERAND = 1 keeps e4m3: both run."""
    eogp_options(score_operand=0 if f4 == "1" else 1)
    rng = np.random.default_rng(N * 7 + Q)
    tc, qc = rand_store(rng, N, ks), rand_store(rng, Q, ks)
    U = len(ks)
    ts = rng.lognormal(0, 0.5, (N, U)).astype(np.float32)
    qs = rng.lognormal(0, 0.5, (Q, U)).astype(np.float32)
    dt = lambda a: torch.from_numpy(a.view(np.int32) if a.dtype == np.uint32 else a).to(DEV)
    out = E.score(dt(tc), dt(ts), ks, E.SCORE_CODES, dt(qc), dt(qs))
    E.sync_status()
    got = out.cpu().numpy()
    want32 = O.score_codes_f32(tc, ts, ks, qc, qs)
    np.testing.assert_array_equal(got, want32)
    want64 = O.score_codes(tc, ts, ks, qc, qs)
    bound = 1e-6 * sum(np.abs(qs[:, u, None] * ts[None, :, u]) * k for u, k in enumerate(ks))
    assert np.all(np.abs(got - want64) <= bound)
    # the tensor-core and popcount kernels agree bit for bit (an empty workspace
    # selects the popcount kernels)
    pop = E.score(dt(tc), dt(ts), ks, E.SCORE_CODES, dt(qc), dt(qs),
                  ws=torch.empty(0, dtype=torch.uint8, device=DEV))
    E.sync_status()
    np.testing.assert_array_equal(pop.cpu().numpy(), got)


@pytest.mark.parametrize("N,Q,ks", [(100, 3, [40, 64, 7]), (257, 70, [1024, 33])])
def test_score_paper_and_fp(N, Q, ks):
    rng = np.random.default_rng(N + Q)
    tc = rand_store(rng, N, ks)
    U, D = len(ks), sum(ks)
    ts = rng.lognormal(0, 0.5, (N, U)).astype(np.float32)
    y = rng.standard_normal((Q, D)).astype(np.float32)
    xt = rng.standard_normal((N, D)).astype(np.float32)
    out = E.score(torch.from_numpy(tc.view(np.int32)).to(DEV), torch.from_numpy(ts).to(DEV), ks,
                  E.SCORE_PAPER, torch.from_numpy(y).to(DEV))
    E.sync_status()
    want = O.score_paper(tc, ts, ks, y)
    scale = sum(np.abs(y[:, None, sum(ks[:u]):sum(ks[:u + 1])]).sum(-1) * ts[None, :, u]
                for u in range(U))
    assert np.all(np.abs(out.cpu().numpy() - want) <= 1e-5 * scale + 1e-30)
    out = E.score(torch.from_numpy(xt).to(DEV), None, ks, E.SCORE_FP, torch.from_numpy(y).to(DEV))
    E.sync_status()
    want = O.score_fp(xt, y)
    scale = np.abs(y) @ np.abs(xt).T
    assert np.all(np.abs(out.cpu().numpy() - want) <= 1e-5 * scale)


# --------------------------------------------------------------- compression

class Layer:
    """One module with synthetic spectra, Haar eigenbases, a, s and a fixed P."""

    def __init__(self, d_in, d_out, T, B, m, k, dtype, alpha=1.2, rel=0.1, seed=0, s_std=0.1,
                 P=None):
        rng = np.random.default_rng(seed)
        rnd = (lambda v: synth.round_to(v, dtype))
        self.QA = rnd(synth.haar_orthogonal(d_in, rng))
        self.QS = rnd(synth.haar_orthogonal(d_out, rng))
        self.lamA = synth.power_spectrum(d_in, alpha)
        self.lamS = synth.power_spectrum(d_out, alpha)
        self.a = rnd(rng.standard_normal((B, T, d_in)))
        self.s = rnd(rng.standard_normal((B, T, d_out)) * s_std)
        self.Pt = rnd(synth.haar_orthogonal(m, rng, k).T) if P is None else rnd(P.T)
        self.m, self.k, self.T, self.B, self.rel = m, k, T, B, rel
        self.dtype = dtype
        self.tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.Lam = O.kfac_eigenvalues(self.lamS, self.lamA)
        self.lam = O.damping(self.Lam, rel)

    def oracle(self):
        z = O.first_stage(self.a, self.s, self.QA, self.QS, self.Lam, self.lam, self.m)
        x = O.project(z, self.Pt.astype(np.float64).T)
        return z, x

    def gpu_desc(self):
        plan = E.Plan.from_factors(self.lamS, self.lamA, self.m, self.rel)
        VA = plan.gather_rows(0, to_dev(self.QA.T, self.tdt))
        VS = plan.gather_rows(1, to_dev(self.QS.T, self.tdt))
        Pt = to_dev(self.Pt, self.tdt)
        self._keep = (plan, VA, VS, Pt)
        return E.layer_desc(plan, self.T, self.k, VA, VS, Pt)

    def gpu_inputs(self):
        return to_dev(self.a, self.tdt), to_dev(self.s, self.tdt)


def run_layer(L, tol):
    desc = L.gpu_desc()
    a, s = L.gpu_inputs()
    z = E.compress_layer(desc, a, s, E.OUT_FIRST_STAGE)
    x = E.compress_layer(desc, a, s, E.OUT_COORDS)
    codes, scales = E.compress_layer(desc, a, s, E.OUT_CODES)
    codes2, scales2 = E.compress_layer(desc, a, s, E.OUT_CODES)
    E.sync_status()
    z_or, x_or = L.oracle()
    rz = row_rel(z.cpu().numpy(), z_or)
    rx = row_rel(x.cpu().numpy(), x_or)
    print(f"[compress] max row rel err z {rz.max():.3e}  x {rx.max():.3e}")
    assert rz.max() <= tol and rx.max() <= tol
    check_bits(x_or, codes_np(codes), L.k)
    _, sc_or = O.onebit(x_or)
    np.testing.assert_allclose(scales.cpu().numpy(), sc_or, rtol=max(tol, 1e-5))
    assert torch.equal(codes, codes2) and torch.equal(scales, scales2)   # deterministic
    return rz.max(), rx.max()


def test_compress_tiny_f32_full_chain():
    """The tiny fp32 workload end to end: 64 -> 64 layer, T = 16, N = 256, m = 512,
    PCA to k = 128 fitted by the oracle on the oracle's z, Q = 8 queries."""
    w = synth.WORKLOADS["tiny_f32"]
    spec = synth.layer_spec(w, 0)
    a, s = synth.layer_inputs(w, 0, w.N)
    Lam = O.kfac_eigenvalues(spec.lam_S, spec.lam_A)
    lam = O.damping(Lam, w.damping_rel)
    z_or = O.first_stage(a, s, spec.Q_A, spec.Q_S, Lam, lam, w.m)
    P, _ = O.fit_pca(z_or, w.k)
    Pt = P.T.astype(np.float32)
    plan = E.Plan.from_factors(spec.lam_S, spec.lam_A, w.m, w.damping_rel)
    VA = plan.gather_rows(0, to_dev(spec.Q_A.T, torch.float32))
    VS = plan.gather_rows(1, to_dev(spec.Q_S.T, torch.float32))
    desc = E.layer_desc(plan, w.T, w.k, VA, VS, to_dev(Pt, torch.float32))
    ad, sd = to_dev(a, torch.float32), to_dev(s, torch.float32)
    z = E.compress_layer(desc, ad, sd, E.OUT_FIRST_STAGE)
    x = E.compress_layer(desc, ad, sd, E.OUT_COORDS)
    codes, scales = E.compress_layer(desc, ad, sd, E.OUT_CODES)
    E.sync_status()
    assert row_rel(z.cpu().numpy(), z_or).max() <= 1e-5
    x_or = O.project(z_or, Pt.astype(np.float64).T)
    assert row_rel(x.cpu().numpy(), x_or).max() <= 1e-5
    check_bits(x_or, codes_np(codes), w.k)
    _, sc_or = O.onebit(x_or)
    np.testing.assert_allclose(scales.cpu().numpy(), sc_or, rtol=1e-5)
    # queries of the same shape, scored against all 256 stored codes
    qa, qs_ = synth.layer_inputs(w, 0, w.Q, role_a=synth.ROLE_QUERY_A, role_s=synth.ROLE_QUERY_S)
    qc, qsc = E.compress_layer(desc, to_dev(qa, torch.float32), to_dev(qs_, torch.float32), E.OUT_CODES)
    sc = E.score(codes, scales[:, None], [w.k], E.SCORE_CODES, qc, qsc[:, None])
    E.sync_status()
    want = O.score_codes_f32(codes_np(codes), scales.cpu().numpy()[:, None], [w.k], codes_np(qc),
                             qsc.cpu().numpy()[:, None])
    np.testing.assert_array_equal(sc.cpu().numpy(), want)


@pytest.mark.parametrize("d_in,d_out,T,B,m,k", [
    (128, 192, 100, 5, 512, 200),    # ragged T (not a multiple of 64) and k
    (64, 64, 64, 3, 1024, 64),       # small square, many retained
    (256, 128, 130, 2, 2000, 130),   # tiles on both axes, odd k
])
def test_compress_bf16_small(d_in, d_out, T, B, m, k):
    L = Layer(d_in, d_out, T, B, m, k, "bf16", seed=d_in + T)
    run_layer(L, 2e-3)


@pytest.mark.parametrize("d_in,d_out", [(768, 2304), (768, 768), (768, 3072), (3072, 768)])
def test_compress_bf16_gpt2_shapes(d_in, d_out):
    """The GPT-2 small module shapes at T = 512, m = 4096, k = 1024."""
    L = Layer(d_in, d_out, 512, 3, 4096, 1024, "bf16", seed=d_in * 7 + d_out)
    rz, rx = run_layer(L, 2e-3)
    assert rx < 1e-4   # the hi/lo split keeps bf16 rounding out of the intermediates


# ------------------------------------------------------------------ fit_pca

def subspace_checks(Pt, eig, Z, k):
    Z64 = Z.astype(np.float64)
    n, m = Z64.shape
    P_or, mu_or = O.fit_pca(Z64, k)
    P = Pt.astype(np.float64).T
    np.testing.assert_allclose(eig, mu_or, rtol=1e-3)
    orth = np.abs(P.T @ P - np.eye(k)).max()
    assert orth <= 1e-4, orth
    C = Z64.T @ Z64 / n
    energy = np.trace(P.T @ C @ P)
    assert energy == pytest.approx(mu_or.sum(), rel=1e-4)
    # principal angles where the eigengap is clear
    allmu = np.sort(np.linalg.eigvalsh(C) if m <= n else np.linalg.eigvalsh(Z64 @ Z64.T / n))[::-1]
    if k < len(allmu) and allmu[k - 1] - allmu[k] > 1e-3 * allmu[0]:
        s = np.linalg.svd(P_or.T @ P, compute_uv=False)
        assert s.min() > 1 - 1e-3


@pytest.mark.parametrize("n,m,k", [(256, 512, 128), (1000, 300, 64), (77, 40, 40),
                                   (1500, 3000, 256),    # subspace solver, Gram route (n < m)
                                   (4000, 2000, 300)])   # subspace solver, covariance route
def test_fit_pca(n, m, k):
    Z = synth.first_stage_like(n, m, seed=n + m)
    Pt, eig = E.fit_pca(torch.from_numpy(Z).to(DEV), k)
    E.sync_status()
    subspace_checks(Pt.cpu().numpy(), eig.cpu().numpy(), Z, k)


@pytest.mark.parametrize("n,m,k", [(1000, 300, 64), (900, 512, 128),
                                   (3000, 1536, 200)])   # subspace solver on the summed moment
def test_fit_pca_from_summed_moments(n, m, k):
    """The sharded fit: second moments of three row shards added on the device
    (accumulate) and the fit from the sum match the oracle like a direct fit."""
    Z = synth.first_stage_like(n, m, seed=n + 2 * m)
    Zd = torch.from_numpy(Z).to(DEV)
    cuts = [0, n // 3, (2 * n) // 3, n]
    C = None
    for a, b in zip(cuts[:-1], cuts[1:]):
        C = E.second_moment(Zd[a:b], C=C, accumulate=C is not None)
    E.sync_status()
    want = Z.astype(np.float64).T @ Z.astype(np.float64)
    np.testing.assert_allclose(C.cpu().numpy(), want, rtol=1e-10, atol=1e-9 * np.abs(want).max())
    Pt, eig = E.fit_pca_from_moment(C, n, k)
    E.sync_status()
    subspace_checks(Pt.cpu().numpy(), eig.cpu().numpy(), Z, k)
    P_or, mu_or = O.fit_pca_from_moment(want, n, k)
    np.testing.assert_allclose(eig.cpu().numpy(), mu_or, rtol=1e-3)


# ------------------------------------------------------------------- errors

def test_workspace_too_small_is_rejected():
    L = Layer(64, 64, 16, 2, 256, 64, "bf16", seed=1)
    desc = L.gpu_desc()
    a, s = L.gpu_inputs()
    need = E.compress_workspace_size(desc, 2, E.OUT_CODES)
    ws = torch.empty(need - 256, dtype=torch.uint8, device=DEV)
    with pytest.raises(E.EOGPError) as ei:
        E.compress_layer(desc, a, s, E.OUT_CODES, ws=ws)
    assert ei.value.code == E.EWORKSPACE


def test_empty_batch_is_a_no_op():
    L = Layer(64, 64, 16, 1, 256, 64, "bf16", seed=2)
    desc = L.gpu_desc()
    a = torch.empty((0, 16, 64), dtype=torch.bfloat16, device=DEV)
    s = torch.empty((0, 16, 64), dtype=torch.bfloat16, device=DEV)
    x = E.compress_layer(desc, a, s, E.OUT_COORDS)
    E.sync_status()
    assert x.shape == (0, 64)
