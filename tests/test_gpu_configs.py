"""GPU parity on every workload shape at full size, on sampled outputs.

* GPT-2 stack: the compression in the exact launch configuration bench.py
  times (B = 512 examples per call, T = 512, m = 4096, k = 1024, device-side
  inputs), checked on sampled examples of one module of each shape.
* OLMo 2 1B / 7B stacks and the 32B gate projection in the launch
  configuration bench.py times (B = 128 / 32 / 64 examples per call, T = 2048,
  m = 8192, k = 2048, device-side inputs): sampled examples of one module of
  each distinct shape, with the oracle's own retained-set selection on the
  full eigenvalue table checked against the plan's sets; and the same shapes
  at B = 1-2 with host-drawn inputs and Haar bases.
* OLMo 2 1B query scoring: Q = 4096 one-bit queries of 112 modules x 2048
  bits against 65,536 stored codes, sampled stored rows bit for bit.
* GPT-2 query scoring: Q = 1024 one-bit queries of 48 modules x 1024 bits
  (the bench's query workload) against 300 stored codes, every score bit for
  bit, dense and with the top-20 ranking fused.
* Scoring sweep: 4,194,304 stored 16,384-bit codes, Q in {1, 64, 1024, 8192};
  sampled stored rows are checked bit for bit.
* PCA fit at the GPT-2 size (10,000 fitting rows, m = 4096, k = 1024) and at
  the OLMo size (10,000 rows, m = 8192, k = 2048).

The oracle is given only the retained eigenvector columns: G~[j, i] for a
retained (j, i) depends on Q_S[:, j] and Q_A[:, i] alone, so restricting Q_A,
Q_S and Lambda to the (ascending) sets C and R changes no retained value and
keeps the canonical order, while the damping still comes from the full table.
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
    torch.cuda.empty_cache()


def oracle_retained(a, s, QA_cols, QS_cols, R, C, Lam_full, lam, m):
    """First-stage z from the retained eigenvector columns only.
    QA_cols [d_in, nC] = Q_A[:, C], QS_cols [d_out, nR] = Q_S[:, R]."""
    Lam_sub = np.asarray(Lam_full)[np.ix_(R, C)]
    return O.first_stage(a, s, QA_cols, QS_cols, Lam_sub, lam, m)


def check_x_codes(x_gpu, codes_gpu, scales_gpu, x_or, k):
    rel = np.linalg.norm(x_gpu - x_or, axis=1) / np.linalg.norm(x_or, axis=1)
    assert rel.max() <= 2e-3, rel.max()
    bits, sc = O.onebit(x_or)
    got = O.unpack_bits(codes_gpu, k)
    small = np.abs(x_or) < 1e-4 * np.linalg.norm(x_or, axis=1, keepdims=True)
    assert not ((got != bits) & ~small).any()
    # the scale is ||x||_1 / k of coordinates held to 2e-3 (bf16 inputs): same bound
    np.testing.assert_allclose(scales_gpu, sc, rtol=2e-3)
    print(f"  max row rel err {rel.max():.2e}; excluded {int(small.sum())}, "
          f"differing there {int(((got != bits) & small).sum())}")
    return rel.max()


# ---------------------------------------------------------------- GPT-2 stack

def test_gpt2_stack_in_bench_launch_configuration():
    import bench
    w = synth.WORKLOADS["gpt2_small_bf16"]
    B = 512
    dev = torch.device(DEV)
    mods = bench.build_stack(w, B, dev, seed=1000)
    ws = E.workspace(max(E.compress_workspace_size(md["desc"], B, E.OUT_CODES) for md in mods), dev)
    words = w.k // 32
    codes = torch.empty((B, len(mods) * words), dtype=torch.int32, device=dev)
    scales = torch.empty((B, len(mods)), dtype=torch.float32, device=dev)
    bench.compress_step(mods, E, codes, scales, ws, words)
    E.sync_status()
    examples = [0, 301, 511]
    for u in (0, 1, 2, 3, 47):    # c_attn, attn.c_proj, c_fc, mlp.c_proj (first block), last module
        md = mods[u]
        desc = md["desc"]
        plan, VA, VS, Pt = desc._refs[:4]
        x = E.compress_layer(desc, md["a"], md["s"], E.OUT_COORDS, ws=ws)
        E.sync_status()
        R, C = plan.sets()
        mod = w.modules[u]
        Lam = O.kfac_eigenvalues(synth.power_spectrum(mod.d_out, w.alpha),
                                 synth.power_spectrum(mod.d_in, w.alpha))
        lam = O.damping(Lam, w.damping_rel)
        a = md["a"][examples].float().cpu().numpy()
        s = md["s"][examples].float().cpu().numpy()
        QA_cols = VA.float().cpu().numpy().T.astype(np.float64)      # [d_in, nC]
        QS_cols = VS.float().cpu().numpy().T.astype(np.float64)      # [d_out, nR]
        z_or = oracle_retained(a, s, QA_cols, QS_cols, R, C, Lam, lam, w.m)
        x_or = O.project(z_or, Pt.float().cpu().numpy().T.astype(np.float64))
        print(f"module {u} ({mod.d_in}->{mod.d_out})")
        check_x_codes(x[examples].cpu().numpy().astype(np.float64),
                      codes[examples, u * words:(u + 1) * words].cpu().numpy().view(np.uint32),
                      scales[examples, u].cpu().numpy(), x_or, w.k)


# ------------------------------------- OLMo / 32B in the bench's launch shape

@pytest.mark.parametrize("name,n_ex", [("olmo2_1b_bf16", 3), ("olmo2_7b_bf16", 2),
                                       ("olmo2_32b_gate_bf16", 3)])
def test_bench_launch_configuration(name, n_ex):
    """One module of each distinct shape compressed exactly as bench.py's
    throughput line launches it (its batch, its inputs, codes written into the
    stack's strided code matrix), checked on n_ex sampled examples against the
    oracle."""
    import bench
    B = bench.CONFIG_BATCH[name]
    dev = torch.device(DEV)
    cs = bench.config_setup(name, B, dev)
    w, per_layer, keys, Pt, descs, ws = (cs[x] for x in ("w", "per_layer", "keys", "Pt", "descs", "ws"))
    words = w.k // 32
    U = len(w.modules)
    codes = torch.empty((B, U * words), dtype=torch.int32, device=dev)
    scales = torch.empty((B, U), dtype=torch.float32, device=dev)
    first = {}
    for u, key in enumerate(keys):
        first.setdefault((key[0], key[1]), u)
    examples = np.linspace(0, B - 1, n_ex).astype(int)
    P = Pt.float().cpu().numpy().T.astype(np.float64)
    for (d_in, d_out), u in first.items():
        key = keys[u]
        L = per_layer[key]
        E.compress_layer(descs[key], L["a"], L["s"], E.OUT_CODES,
                         codes=codes[:, u * words:(u + 1) * words], scales=scales[:, u], ws=ws)
        x = E.compress_layer(descs[key], L["a"], L["s"], E.OUT_COORDS, ws=ws)
        E.sync_status()
        if w.spectrum == "channel":
            sp = synth.layer_spec(w, u, 1, 1)
            lamA, lamS = sp.lam_A, sp.lam_S
        else:
            lamA, lamS = synth.power_spectrum(d_in, w.alpha), synth.power_spectrum(d_out, w.alpha)
        Lam = O.kfac_eigenvalues(lamS, lamA)
        lam = O.damping(Lam, w.damping_rel)
        # the oracle's own top-m selection on the full table gives the plan's sets
        j_or, i_or = O.select_retained(Lam, w.m)
        R, C = L["plan"].sets()
        np.testing.assert_array_equal(R, np.unique(j_or))
        np.testing.assert_array_equal(C, np.unique(i_or))
        a = L["a"][examples].float().cpu().numpy()
        s_ = L["s"][examples].float().cpu().numpy()
        QA_cols = L["VA"].float().cpu().numpy().T.astype(np.float64)
        QS_cols = L["VS"].float().cpu().numpy().T.astype(np.float64)
        z_or = oracle_retained(a, s_, QA_cols, QS_cols, R, C, Lam, lam, w.m)
        x_or = O.project(z_or, P)
        print(f"{name} module {u} ({d_in}->{d_out}) B={B} examples {list(examples)}")
        check_x_codes(x[examples].cpu().numpy().astype(np.float64),
                      codes[examples, u * words:(u + 1) * words].cpu().numpy().view(np.uint32),
                      scales[examples, u].cpu().numpy(), x_or, w.k)
        del x
    del cs, per_layer, descs, ws, codes, scales
    torch.cuda.empty_cache()


# --------------------------------------------------------- OLMo-shaped layers

def run_shape(w, u, B, seed):
    mod = w.modules[u]
    spec_lam = synth.layer_spec(w, u, 1, 1) if w.spectrum == "channel" else None
    if w.spectrum == "channel":
        lamA, lamS = spec_lam.lam_A, spec_lam.lam_S
    else:
        lamA, lamS = synth.power_spectrum(mod.d_in, w.alpha), synth.power_spectrum(mod.d_out, w.alpha)
    plan = E.Plan.from_factors(lamS, lamA, w.m, w.damping_rel)
    inf = plan.info()
    R, C = plan.sets()
    # Retained eigenvector columns (full bases are d x d; only these are read).
    if w.spectrum == "channel":
        full = synth.layer_spec(w, u)
        QA_cols, QS_cols = full.Q_A[:, C], full.Q_S[:, R]
        chan = full
    else:
        assert (C == np.arange(inf.nC)).all() and (R == np.arange(inf.nR)).all()
        sp = synth.layer_spec(w, u, inf.nC, inf.nR)
        QA_cols, QS_cols = sp.Q_A, sp.Q_S
        chan = None
    rng = np.random.default_rng(seed)
    Pt = np.ascontiguousarray(synth.round_bf16(synth.haar_orthogonal(w.m, rng, w.k).T))
    a, s = synth.layer_inputs(w, u, B, spec=chan)
    bf = torch.bfloat16
    VA = torch.from_numpy(np.ascontiguousarray(QA_cols.T)).to(DEV, bf)
    VS = torch.from_numpy(np.ascontiguousarray(QS_cols.T)).to(DEV, bf)
    desc = E.layer_desc(plan, w.T, w.k, VA, VS, torch.from_numpy(Pt).to(DEV, bf))
    ad, sd = torch.from_numpy(a).to(DEV, bf), torch.from_numpy(s).to(DEV, bf)
    x = E.compress_layer(desc, ad, sd, E.OUT_COORDS)
    codes, scales = E.compress_layer(desc, ad, sd, E.OUT_CODES)
    E.sync_status()
    Lam = O.kfac_eigenvalues(lamS, lamA)
    lam = O.damping(Lam, w.damping_rel)
    z_or = oracle_retained(a, s, QA_cols.astype(np.float64), QS_cols.astype(np.float64), R, C,
                           Lam, lam, w.m)
    x_or = O.project(z_or, Pt.astype(np.float64).T)
    print(f"{w.name} module {u} ({mod.d_in}->{mod.d_out}) nR={inf.nR} nC={inf.nC} "
          f"tiles={inf.n_tiles}")
    check_x_codes(x.cpu().numpy().astype(np.float64), codes.cpu().numpy().view(np.uint32),
                  scales.cpu().numpy(), x_or, w.k)


@pytest.mark.parametrize("u", [0, 4, 6])   # q_proj 2048x2048, gate 2048->8192, down 8192->2048
def test_olmo2_1b_shapes(u):
    run_shape(synth.WORKLOADS["olmo2_1b_bf16"], u, 2, seed=31 + u)


@pytest.mark.parametrize("u", [0, 4, 6])   # 4096x4096, gate 4096->11008, down 11008->4096
def test_olmo2_7b_shapes(u):
    run_shape(synth.WORKLOADS["olmo2_7b_bf16"], u, 1, seed=71 + u)


def test_olmo2_32b_gate():
    run_shape(synth.WORKLOADS["olmo2_32b_gate_bf16"], 0, 1, seed=32)


# ------------------------------------------------------------- scoring sweep

@pytest.mark.parametrize("Q", [1, 64, 1024, 8192])
def test_scan_sweep_sampled_rows(Q):
    sc = synth.SCAN
    N, k = sc["N"], sc["k"]
    W = k // 32
    g = torch.Generator(device=DEV)
    g.manual_seed(sc["seed"])
    train = torch.randint(-2 ** 31, 2 ** 31 - 1, (N, W), generator=g, device=DEV, dtype=torch.int32)
    tsc = torch.exp(sc["scale_sigma"] * torch.randn((N, 1), generator=g, device=DEV))
    query = torch.randint(-2 ** 31, 2 ** 31 - 1, (Q, W), generator=g, device=DEV, dtype=torch.int32)
    qsc = torch.exp(sc["scale_sigma"] * torch.randn((Q, 1), generator=g, device=DEV))
    rows = np.arange(0, N, 65537 if Q >= 1024 else 4099)
    qchunk = 1024
    for q0 in range(0, Q, qchunk):
        q1 = min(Q, q0 + qchunk)
        out = E.score(train, tsc, [k], E.SCORE_CODES, query[q0:q1], qsc[q0:q1])
        E.sync_status()
        got = out[:, rows].cpu().numpy()
        qsel = slice(0, q1 - q0) if Q <= 64 else np.arange(0, q1 - q0, 97)
        tr = train[rows].cpu().numpy().view(np.uint32)
        qc = query[q0:q1].cpu().numpy().view(np.uint32)[qsel]
        want = O.score_codes_f32(tr, tsc[rows].cpu().numpy(), [k], qc,
                                 qsc[q0:q1].cpu().numpy()[qsel])
        np.testing.assert_array_equal(got[qsel], want)
        del out
    del train, query
    torch.cuda.empty_cache()


# ------------------------------------------------- OLMo-1B query scoring

def test_olmo2_1b_query_scoring_sampled_rows():
    """Q = 4096 one-bit queries of 112 modules x 2048 bits (the OLMo-1B stack's
    codes) against 65,536 stored codes: every score of 16 sampled stored rows
    equals the oracle's float32 evaluation bit for bit."""
    w = synth.WORKLOADS["olmo2_1b_bf16"]
    U, k = len(w.modules), w.k
    ks = [k] * U
    N, Q = 65536, w.Q
    W = U * k // 32
    g = torch.Generator(device=DEV)
    g.manual_seed(4096)
    train = torch.randint(-2 ** 31, 2 ** 31 - 1, (N, W), generator=g, device=DEV, dtype=torch.int32)
    query = torch.randint(-2 ** 31, 2 ** 31 - 1, (Q, W), generator=g, device=DEV, dtype=torch.int32)
    tsc = torch.exp(0.5 * torch.randn((N, U), generator=g, device=DEV))
    qsc = torch.exp(0.5 * torch.randn((Q, U), generator=g, device=DEV))
    out = E.score(train, tsc, ks, E.SCORE_CODES, query, qsc)
    E.sync_status()
    rows = np.arange(0, N, 4099)
    got = out[:, rows].cpu().numpy()
    del out
    want = O.score_codes_f32(train[rows].cpu().numpy().view(np.uint32), tsc[rows].cpu().numpy(), ks,
                             query.cpu().numpy().view(np.uint32), qsc.cpu().numpy())
    np.testing.assert_array_equal(got, want)
    del train, query
    torch.cuda.empty_cache()


# -------------------------------------------------------------------- PCA fit

def test_fit_pca_gpt2_size():
    n, m, k = 10000, 4096, 1024
    Z = synth.first_stage_like(n, m, seed=5)
    Pt, eig = E.fit_pca(torch.from_numpy(Z).to(DEV), k)
    E.sync_status()
    P = Pt.cpu().numpy().astype(np.float64).T
    Z64 = Z.astype(np.float64)
    C = Z64.T @ Z64 / n
    mu = np.sort(np.linalg.eigvalsh(C))[::-1]
    np.testing.assert_allclose(eig.cpu().numpy(), mu[:k], rtol=1e-3)
    assert np.abs(P.T @ P - np.eye(k)).max() <= 1e-4
    assert np.trace(P.T @ C @ P) == pytest.approx(mu[:k].sum(), rel=1e-4)


# ------------------------------------------------------ GPT-2 query scoring

def test_gpt2_query_scoring_all_scores(eogp_options):
    """Q = 1024 queries x 48 modules x 1024 bits (the bench's query workload: the
    running score kept in TMEM across modules) against N = 300 stored codes (a
    ragged last row tile): every score equals the oracle's float32 evaluation
    bit for bit, and the fused top-20 equals the oracle ranking."""
    rng = np.random.default_rng(48)
    ks = [1024] * 48
    N, Q = 300, 1024
    W = sum(ks) // 32
    tc = rng.integers(0, 2**32, (N, W), dtype=np.uint64).astype(np.uint32)
    qc = rng.integers(0, 2**32, (Q, W), dtype=np.uint64).astype(np.uint32)
    ts = rng.lognormal(0, 0.5, (N, 48)).astype(np.float32)
    qs = rng.lognormal(0, 0.5, (Q, 48)).astype(np.float32)
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(DEV)
    tcd, qcd = d(tc.view(np.int32)), d(qc.view(np.int32))
    want = O.score_codes_f32(tc, ts, ks, qc, qs)
    want_v, want_i = O.top_k(want, 20)
    for f4 in ("1", "0"):            # e2m1 operands (the default here) and e4m3
        eogp_options(score_operand=0 if f4 == "1" else 1)
        got = E.score(tcd, d(ts), ks, E.SCORE_CODES, qcd, d(qs))
        E.sync_status()
        np.testing.assert_array_equal(got.cpu().numpy(), want)
        for fused in ("1", "0"):     # ranking fused into the scoring kernel, and the dense path
            eogp_options(topk_path=1 if fused == "1" else 2)
            vals, idx = E.score_topk(tcd, d(ts), ks, E.SCORE_CODES, qcd, 20, query_scales=d(qs))
            E.sync_status()
            np.testing.assert_array_equal(idx.cpu().numpy(), want_i)
            np.testing.assert_array_equal(vals.cpu().numpy().astype(np.float64), want_v)


def test_fit_pca_olmo_size():
    """The fit at the OLMo workloads' size: 10,000 fitting rows, m = 8192, k = 2048."""
    from test_gpu_parity import subspace_checks
    n, m, k = 10000, 8192, 2048
    Z = synth.first_stage_like(n, m, seed=6)
    Pt, eig = E.fit_pca(torch.from_numpy(Z).to(DEV), k)
    E.sync_status()
    subspace_checks(Pt.cpu().numpy(), eig.cpu().numpy(), Z, k)
