"""GPU parity of paper-mode tensor-core scoring and of the per-query ranking.

* PAPER mode on the tensor cores (y split into bf16 hi + lo, bits expanded to
  +-1) against the oracle's float64 sum_u s_iu <y_u, b_iu>, within
  1e-5 * sum_u s_iu ||y_u||_1, and against the CUDA-core kernel.
* eogp_score_topk against the oracle's ranking: CODES scores are bitwise
  reproducible, so the lists must match exactly (values and indices, including
  planted equal scores); PAPER / FP lists are checked for validity within the
  score tolerance (several lists are correct when scores differ by less).
* The three paths: up to 49,152 stored rows, dense scores and a radix select
  per query row (the library's choice there); beyond, the ranking fused into
  the tensor-core epilogue (K <= 32), else dense scores, per-slot lists and a
  merge. EOGP_OPT_TOPK_PATH = 1 / 2 forces the fused / a dense path, which the
  tests use to run both on the same cases; edge cases N < K and N = 0, ties.
* Full scan scale (4,194,304 stored 16,384-bit codes, Q = 1024): the fused
  lists equal the oracle ranking of the dense scores of sampled queries.
"""
import numpy as np
import pytest

from oracle import eogp_oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2609_37842_gb300 import eogp as E  # noqa: E402
from paper_2609_37842_gb300 import synth  # noqa: E402

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_37842_gb300 import build
    build.build()
    E.lib()
    yield
    torch.cuda.empty_cache()


def rand_store(rng, n, ks):
    return O.pack_concat([rng.integers(0, 2, (n, k)).astype(bool) for k in ks])


def dev(a):
    return torch.from_numpy(a.view(np.int32) if a.dtype == np.uint32 else a).to(DEV)


def paper_scale(y, ts, ks):
    """sum_u s_iu ||y_qu||_1 -> [Q, N]: the magnitude the PAPER tolerance is relative to."""
    off = np.cumsum([0] + list(ks))
    return sum(np.abs(y[:, off[u]:off[u + 1]]).sum(1)[:, None] * ts[None, :, u].astype(np.float64)
               for u in range(len(ks)))


def check_valid_topk(vals, idx, S, tol, K):
    """(vals, idx) is a correct top-K of the exact scores S [Q, N] when scores are
    known only to +-tol [Q, N]: values match their rows, are sorted, rows are
    distinct, and no omitted row beats an included one by more than the tolerance."""
    Q, N = S.shape
    kk = min(K, N)
    assert (idx[:, kk:] == -1).all() and np.isneginf(vals[:, kk:]).all()
    for q in range(Q):
        i = idx[q, :kk]
        assert len(set(i.tolist())) == kk and i.min() >= 0 and i.max() < N
        assert np.all(np.abs(vals[q, :kk] - S[q, i]) <= tol[q, i])
        assert np.all(np.diff(vals[q, :kk]) <= 0)
        rest = np.setdiff1d(np.arange(N), i)
        if len(rest):
            worst_in = np.min(S[q, i] + tol[q, i])
            assert np.all(S[q, rest] - tol[q, rest] <= worst_in)


# ------------------------------------------------------------ paper, dense

@pytest.mark.parametrize("N,Q,ks", [(1000, 70, [64, 128, 192]), (300, 1, [1024]),
                                    (2000, 130, [1024] * 6), (129, 257, [64])])
def test_score_paper_tensor_cores(N, Q, ks):
    rng = np.random.default_rng(N + 3 * Q)
    tc = rand_store(rng, N, ks)
    ts = rng.lognormal(0, 0.5, (N, len(ks))).astype(np.float32)
    y = (rng.standard_normal((Q, sum(ks))) * rng.lognormal(0, 1, (1, sum(ks)))).astype(np.float32)
    out = E.score(dev(tc), dev(ts), ks, E.SCORE_PAPER, dev(y))
    E.sync_status()
    got = out.cpu().numpy().astype(np.float64)
    want = O.score_paper(tc, ts, ks, y)
    scale = paper_scale(y, ts, ks)
    err = np.abs(got - want) / scale
    print(f"max |err| / (sum_u s ||y||_1) = {err.max():.2e}")
    assert err.max() <= 1e-5
    simt = E.score(dev(tc), dev(ts), ks, E.SCORE_PAPER, dev(y), ws=torch.empty(0, dtype=torch.uint8, device=DEV))
    E.sync_status()
    assert np.all(np.abs(simt.cpu().numpy() - want) <= 1e-5 * scale)


# ------------------------------------------------------------ ranking

def codes_case(N, Q, ks, seed, dup=True):
    rng = np.random.default_rng(seed)
    tc, qc = rand_store(rng, N, ks), rand_store(rng, Q, ks)
    ts = rng.lognormal(0, 0.5, (N, len(ks))).astype(np.float32)
    qs = rng.lognormal(0, 0.5, (Q, len(ks))).astype(np.float32)
    if dup and N >= 40:
        # planted equal scores: stored rows repeated further down the store
        h = N // 4
        tc[N - h:] = tc[:h]
        ts[N - h:] = ts[:h]
    return tc, ts, qc, qs


@pytest.mark.parametrize("N,Q,ks,K", [(1000, 70, [128, 256], 10), (5000, 130, [1024, 1024], 32),
                                      (300, 64, [128], 1), (20, 64, [128], 32),
                                      (20000, 200, [512], 20), (30000, 300, [1024], 20),
                                      (3000, 300, [512, 1024, 128], 20),   # several modules, two query tiles
                                      (5000, 130, [1024, 1024], 64)])
@pytest.mark.parametrize("fused", ["1", "0"])
@pytest.mark.parametrize("f4", ["1", "0"])
def test_topk_codes_fused_exact(N, Q, ks, K, fused, f4, eogp_options):
    """K <= 32 ranks inside the tensor-core epilogue when fused; K = 64 always
    takes the dense path. Both paths give the oracle's lists exactly, with e2m1
    operands (modules of multiples of 256 bits) and with e4m3 (EOGP_OPT_SCORE_OPERAND = 1)."""
    eogp_options(topk_path=1 if fused == "1" else 2)
    eogp_options(score_operand=0 if f4 == "1" else 1)
    tc, ts, qc, qs = codes_case(N, Q, ks, N + K)
    vals, idx = E.score_topk(dev(tc), dev(ts), ks, E.SCORE_CODES, dev(qc), K, query_scales=dev(qs))
    E.sync_status()
    want_v, want_i = O.top_k(O.score_codes_f32(tc, ts, ks, qc, qs), K)
    np.testing.assert_array_equal(idx.cpu().numpy(), want_i)
    np.testing.assert_array_equal(vals.cpu().numpy().astype(np.float64), want_v)


@pytest.mark.parametrize("N,Q,ks,K", [(3000, 5, [128, 64], 16), (4000, 70, [256], 100),
                                      (700, 33, [1024], 256),
                                      (60000, 33, [128], 100),      # beyond the select: slot lists + merge
                                      (50000, 70, [256, 128], 40)])
def test_topk_codes_dense_exact(N, Q, ks, K):
    tc, ts, qc, qs = codes_case(N, Q, ks, N + K + 1)
    vals, idx = E.score_topk(dev(tc), dev(ts), ks, E.SCORE_CODES, dev(qc), K, query_scales=dev(qs))
    E.sync_status()
    want_v, want_i = O.top_k(O.score_codes_f32(tc, ts, ks, qc, qs), K)
    np.testing.assert_array_equal(idx.cpu().numpy(), want_i)
    np.testing.assert_array_equal(vals.cpu().numpy().astype(np.float64), want_v)


@pytest.mark.parametrize("N,Q,ks,K", [(1500, 70, [64, 128], 20), (4000, 3, [256], 10),
                                      (600, 130, [128], 100)])
@pytest.mark.parametrize("fused", ["1", "0"])
def test_topk_paper_valid(N, Q, ks, K, fused, eogp_options):
    eogp_options(topk_path=1 if fused == "1" else 2)
    rng = np.random.default_rng(N + Q + K)
    tc = rand_store(rng, N, ks)
    ts = rng.lognormal(0, 0.5, (N, len(ks))).astype(np.float32)
    y = rng.standard_normal((Q, sum(ks))).astype(np.float32)
    vals, idx = E.score_topk(dev(tc), dev(ts), ks, E.SCORE_PAPER, dev(y), K)
    E.sync_status()
    S = O.score_paper(tc, ts, ks, y)
    check_valid_topk(vals.cpu().numpy().astype(np.float64), idx.cpu().numpy(), S,
                     1e-5 * paper_scale(y, ts, ks), K)


def test_topk_fp_valid():
    rng = np.random.default_rng(5)
    N, Q, D, K = 900, 40, 96, 12
    xt = rng.standard_normal((N, D)).astype(np.float32)
    y = rng.standard_normal((Q, D)).astype(np.float32)
    vals, idx = E.score_topk(dev(xt), None, [D], E.SCORE_FP, dev(y), K)
    E.sync_status()
    S = O.score_fp(xt, y)
    check_valid_topk(vals.cpu().numpy().astype(np.float64), idx.cpu().numpy(), S,
                     1e-5 * (np.abs(y) @ np.abs(xt).T), K)


def test_topk_empty_store():
    qc = rand_store(np.random.default_rng(0), 70, [128])
    qs = np.ones((70, 1), np.float32)
    tc = np.zeros((0, 4), np.uint32)
    ts = np.zeros((0, 1), np.float32)
    vals, idx = E.score_topk(dev(tc), dev(ts), [128], E.SCORE_CODES, dev(qc), 5, query_scales=dev(qs))
    E.sync_status()
    assert (idx.cpu().numpy() == -1).all() and np.isneginf(vals.cpu().numpy()).all()


def test_topk_scan_scale_sampled_queries():
    sc = synth.SCAN
    N, k, Q, K = sc["N"], sc["k"], 1024, 20
    W = k // 32
    g = torch.Generator(device=DEV)
    g.manual_seed(sc["seed"])
    train = torch.randint(-2 ** 31, 2 ** 31 - 1, (N, W), generator=g, device=DEV, dtype=torch.int32)
    tsc = torch.exp(sc["scale_sigma"] * torch.randn((N, 1), generator=g, device=DEV))
    query = torch.randint(-2 ** 31, 2 ** 31 - 1, (Q, W), generator=g, device=DEV, dtype=torch.int32)
    qsc = torch.exp(sc["scale_sigma"] * torch.randn((Q, 1), generator=g, device=DEV))
    vals, idx = E.score_topk(train, tsc, [k], E.SCORE_CODES, query, K, query_scales=qsc)
    E.sync_status()
    qsel = [0, 1, 127, 128, 513, 1023]
    dense = E.score(train, tsc, [k], E.SCORE_CODES, query[qsel], qsc[qsel])
    E.sync_status()
    dn = dense.cpu().numpy()
    want_v, want_i = O.top_k(dn, K)
    np.testing.assert_array_equal(idx[qsel].cpu().numpy(), want_i)
    np.testing.assert_array_equal(vals[qsel].cpu().numpy().astype(np.float64), want_v)
    # the dense scores behind the comparison are the oracle's: on sampled stored
    # rows by explicit +-1 sums, and on every stored row by the XOR / population
    # count form, in the same float32 order (one module: fl(fl(s_q s_i) d))
    rows = np.unique(np.concatenate([want_i.reshape(-1), np.arange(0, N, 524287)]))
    tr = train[rows].cpu().numpy().view(np.uint32)
    ref = O.score_codes_f32(tr, tsc[rows].cpu().numpy(), [k], query[qsel].cpu().numpy().view(np.uint32),
                            qsc[qsel].cpu().numpy())
    np.testing.assert_array_equal(dn[:, rows], ref)
    qh = query[qsel].cpu().numpy().view(np.uint32)
    qsh = qsc[qsel].cpu().numpy()[:, 0]
    ts_all = tsc.cpu().numpy()[:, 0]
    step = 1 << 18
    for r0 in range(0, N, step):
        tw = train[r0:r0 + step].cpu().numpy().view(np.uint32)
        for j in range(len(qsel)):
            d = O.onebit_dot_xor(tw, qh[j], k).astype(np.float32)
            sp = (qsh[j] * ts_all[r0:r0 + step]).astype(np.float32)
            np.testing.assert_array_equal(dn[j, r0:r0 + step], (sp * d).astype(np.float32))
    del train, query, dense
    torch.cuda.empty_cache()
