"""GPU parity of the real-workload plumbing of the compression call against
the oracle: a module bias as a constant-1 input channel (App. C.1, GPT-2
attributes biases) and variable-length examples padded to T (App. C.1,
conversations of at most 2048 tokens), separately and together, on the bf16
tensor-core path (within 2e-3 per row) and the fp32 path (within 1e-5).
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


def dev(a, dt=None):
    t = torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    return t.to(dt) if dt is not None else t


def row_rel(got, want):
    return np.linalg.norm(got - want, axis=1) / np.linalg.norm(want, axis=1)


@pytest.mark.parametrize("dtype,d_in,d_out,T,B,m,k,bias,lens,tol", [
    ("bf16", 768, 768, 100, 4, 4096, 1024, True, False, 2e-3),
    ("bf16", 256, 384, 128, 5, 2000, 300, False, True, 2e-3),
    ("bf16", 768, 2304, 130, 3, 4096, 1024, True, True, 2e-3),
    ("f32", 64, 64, 16, 6, 512, 128, True, True, 1e-5),
])
def test_bias_and_lengths(dtype, d_in, d_out, T, B, m, k, bias, lens, tol):
    rng = np.random.default_rng(d_in + T + B)
    rnd = (lambda v: synth.round_to(v, dtype))
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    d_eff = d_in + (1 if bias else 0)
    QA, QS = rnd(synth.haar_orthogonal(d_eff, rng)), rnd(synth.haar_orthogonal(d_out, rng))
    lamA, lamS = synth.power_spectrum(d_eff, 1.2), synth.power_spectrum(d_out, 1.2)
    a = rnd(rng.standard_normal((B, T, d_in)))
    s = rnd(rng.standard_normal((B, T, d_out)) * 0.1)
    lengths = rng.integers(1, T + 1, B).astype(np.int32) if lens else None
    if lens:
        lengths[0] = T          # one full example, and one cut very short
        lengths[-1] = 1
    Pt = rnd(synth.haar_orthogonal(m, rng, k).T)
    plan = E.Plan.from_factors(lamS, lamA, m, 0.1)
    R, C = plan.sets()
    VA_full = QA.T[C]                       # [nC, d_eff]: retained eigenvectors as rows
    VA = np.ascontiguousarray(VA_full[:, :d_in], dtype=np.float32)
    bias_A = np.ascontiguousarray(VA_full[:, d_in], dtype=np.float32) if bias else None
    VS = np.ascontiguousarray(QS.T[R], dtype=np.float32)
    desc = E.layer_desc(plan, T, k, dev(VA, tdt), dev(VS, tdt), dev(Pt.astype(np.float32), tdt),
                        bias_A=dev(bias_A) if bias else None,
                        lengths=dev(lengths) if lens else None)
    ad, sd = dev(a.astype(np.float32), tdt), dev(s.astype(np.float32), tdt)
    x = E.compress_layer(desc, ad, sd, E.OUT_COORDS)
    codes, scales = E.compress_layer(desc, ad, sd, E.OUT_CODES)
    E.sync_status()
    a_or = O.with_bias_channel(a) if bias else a
    s_or = O.mask_tokens(s, lengths) if lens else s
    Lam = O.kfac_eigenvalues(lamS, lamA)
    z_or = O.first_stage(a_or, s_or, QA, QS, Lam, O.damping(Lam, 0.1), m)
    x_or = O.project(z_or, Pt.astype(np.float64).T)
    rel = row_rel(x.cpu().numpy().astype(np.float64), x_or)
    print(f"max row rel err {rel.max():.2e}")
    assert rel.max() <= tol
    bits, sc = O.onebit(x_or)
    got = O.unpack_bits(codes.cpu().numpy().view(np.uint32), k)
    small = np.abs(x_or) < 1e-4 * np.linalg.norm(x_or, axis=1, keepdims=True)
    assert not ((got != bits) & ~small).any()
    np.testing.assert_allclose(scales.cpu().numpy(), sc, rtol=max(tol, 1e-5))
    if bias:   # the bias channel changes the result (the term is really used)
        z_nob = O.first_stage(np.concatenate([a, np.zeros(a.shape[:-1] + (1,))], -1), s_or, QA, QS,
                              Lam, O.damping(Lam, 0.1), m)
        assert row_rel(O.project(z_nob, Pt.astype(np.float64).T), x_or).min() > 10 * rel.max()


@pytest.mark.parametrize("N,ks", [(37, [13, 32, 70]), (300, [1024] * 48), (1, [1])])
def test_store_records(N, ks, tmp_path):
    """Store records (App. E.1): bytes equal the oracle's, the round trip gives the
    codes back and the scales rounded to half precision, and a file written and
    read back scores exactly like the records it came from."""
    rng = np.random.default_rng(N + len(ks))
    codes = O.pack_concat([rng.integers(0, 2, (N, k)).astype(bool) for k in ks])
    scales = rng.lognormal(0, 0.5, (N, len(ks))).astype(np.float32)
    cd, sd = dev(codes.view(np.int32)), dev(scales)
    pay = E.payload_pack(cd, sd, ks)
    E.sync_status()
    want = O.to_payload(codes, scales, ks)
    assert pay.shape[1] == O.payload_bytes(ks)
    np.testing.assert_array_equal(pay.cpu().numpy(), want)
    c2, s2 = E.payload_unpack(pay, ks)
    E.sync_status()
    wc, ws = O.from_payload(want, ks)
    np.testing.assert_array_equal(c2.cpu().numpy().view(np.uint32), wc)
    np.testing.assert_array_equal(s2.cpu().numpy(), ws)
    path = str(tmp_path / "store.bin")
    E.write_store(path, pay)
    back = E.read_store(path, ks, DEV)
    assert torch.equal(back, pay)
    if all(k % 32 == 0 for k in ks):
        q = min(N, 5)
        sc = E.score(c2, s2, ks, E.SCORE_CODES, c2[:q], s2[:q])
        E.sync_status()
        np.testing.assert_array_equal(sc.cpu().numpy(), O.score_codes_f32(wc, ws, ks, wc[:q], ws[:q]))


def test_host_resident_eigenbases_give_identical_codes():
    """Eigenvector rows in page-locked host memory (copied by each call) give the
    same results, bit for bit, as device-resident ones."""
    rng = np.random.default_rng(13)
    d_in, d_out, T, B, m, k = 768, 768, 64, 3, 4096, 1024
    QA = synth.round_to(synth.haar_orthogonal(d_in, rng), "bf16")
    QS = synth.round_to(synth.haar_orthogonal(d_out, rng), "bf16")
    plan = E.Plan.from_factors(synth.power_spectrum(d_out, 1.2), synth.power_spectrum(d_in, 1.2), m, 0.1)
    R, C = plan.sets()
    VA = torch.from_numpy(np.ascontiguousarray(QA.T[C], dtype=np.float32)).to(torch.bfloat16)
    VS = torch.from_numpy(np.ascontiguousarray(QS.T[R], dtype=np.float32)).to(torch.bfloat16)
    Pt = dev(synth.round_to(synth.haar_orthogonal(m, rng, k).T, "bf16").astype(np.float32), torch.bfloat16)
    a = dev(synth.round_to(rng.standard_normal((B, T, d_in)), "bf16").astype(np.float32), torch.bfloat16)
    s = dev(synth.round_to(rng.standard_normal((B, T, d_out)) * 0.1, "bf16").astype(np.float32), torch.bfloat16)
    d_dev = E.layer_desc(plan, T, k, VA.to(DEV), VS.to(DEV), Pt)
    d_host = E.layer_desc(plan, T, k, VA.pin_memory(), VS.pin_memory(), Pt)
    c1, s1 = E.compress_layer(d_dev, a, s, E.OUT_CODES)
    c2, s2 = E.compress_layer(d_host, a, s, E.OUT_CODES)
    x1 = E.compress_layer(d_dev, a, s, E.OUT_COORDS)
    x2 = E.compress_layer(d_host, a, s, E.OUT_COORDS)
    E.sync_status()
    assert torch.equal(c1, c2) and torch.equal(s1, s2) and torch.equal(x1, x2)


@pytest.mark.parametrize("dtype,d_in,d_out,T,B,m,k,chunk,bias,lens,host_bases", [
    ("bf16", 768, 2304, 64, 7, 4096, 1024, 3, True, True, False),
    ("bf16", 768, 768, 64, 5, 4096, 1024, 0, False, False, True),
    ("bf16", 256, 384, 128, 4, 2000, 300, 1, False, True, True),
    ("f32", 64, 64, 16, 9, 512, 128, 4, True, False, False),
])
def test_host_inputs_match_device_inputs(dtype, d_in, d_out, T, B, m, k, chunk, bias, lens, host_bases):
    """eogp_compress_layer_host (inputs in page-locked host memory, copied chunk by
    chunk by the call) gives the results of eogp_compress_layer on the same
    inputs in device memory, bit for bit, in every output mode: ragged last
    chunk, per-example lengths offset per chunk, bias channel, host eigenbases."""
    rng = np.random.default_rng(d_in + B + chunk)
    rnd = (lambda v: synth.round_to(v, dtype))
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    d_eff = d_in + (1 if bias else 0)
    QA, QS = rnd(synth.haar_orthogonal(d_eff, rng)), rnd(synth.haar_orthogonal(d_out, rng))
    plan = E.Plan.from_factors(synth.power_spectrum(d_out, 1.2), synth.power_spectrum(d_eff, 1.2), m, 0.1)
    R, C = plan.sets()
    VA_full = QA.T[C]
    VA = torch.from_numpy(np.ascontiguousarray(VA_full[:, :d_in], dtype=np.float32)).to(tdt)
    VS = torch.from_numpy(np.ascontiguousarray(QS.T[R], dtype=np.float32)).to(tdt)
    if host_bases:
        VA, VS = VA.pin_memory(), VS.pin_memory()
    else:
        VA, VS = VA.to(DEV), VS.to(DEV)
    bias_A = dev(np.ascontiguousarray(VA_full[:, d_in], dtype=np.float32)) if bias else None
    lengths = None
    if lens:
        lv = rng.integers(1, T + 1, B).astype(np.int32)
        lv[0] = T
        lengths = dev(lv)
    Pt = dev(rnd(synth.haar_orthogonal(m, rng, k).T).astype(np.float32), tdt)
    desc = E.layer_desc(plan, T, k, VA, VS, Pt, bias_A=bias_A, lengths=lengths)
    a = torch.from_numpy(rnd(rng.standard_normal((B, T, d_in))).astype(np.float32)).to(tdt)
    s = torch.from_numpy(rnd(rng.standard_normal((B, T, d_out)) * 0.1).astype(np.float32)).to(tdt)
    if chunk == 3:      # inputs in eogp_host_alloc memory
        ah, sh = E.host_empty(a.shape, tdt), E.host_empty(s.shape, tdt)
        ah.copy_(a)
        sh.copy_(s)
    else:
        ah, sh = a.pin_memory(), s.pin_memory()
    ad, sd = a.to(DEV), s.to(DEV)
    c1, s1 = E.compress_layer(desc, ad, sd, E.OUT_CODES)
    c2, s2 = E.compress_layer_host(desc, ah, sh, E.OUT_CODES, DEV, chunk=chunk)
    for mode in (E.OUT_COORDS, E.OUT_FIRST_STAGE):
        x1 = E.compress_layer(desc, ad, sd, mode)
        x2 = E.compress_layer_host(desc, ah, sh, mode, DEV, chunk=chunk)
        torch.cuda.synchronize()
        assert torch.equal(x1, x2), mode
    E.sync_status()
    assert torch.equal(c1, c2) and torch.equal(s1, s2)


def _host_module(rng, d_in, d_out, T, m, k, host_bases, lengths=None):
    """One bf16 module: plan, descriptor, its own inputs (host and device)."""
    rnd = (lambda v: synth.round_to(v, "bf16"))
    tdt = torch.bfloat16
    QA, QS = rnd(synth.haar_orthogonal(d_in, rng)), rnd(synth.haar_orthogonal(d_out, rng))
    plan = E.Plan.from_factors(synth.power_spectrum(d_out, 1.2), synth.power_spectrum(d_in, 1.2), m, 0.1)
    R, C = plan.sets()
    VA = torch.from_numpy(np.ascontiguousarray(QA.T[C], dtype=np.float32)).to(tdt)
    VS = torch.from_numpy(np.ascontiguousarray(QS.T[R], dtype=np.float32)).to(tdt)
    if host_bases:
        hva, hvs = E.host_empty(VA.shape, tdt), E.host_empty(VS.shape, tdt)
        hva.copy_(VA)
        hvs.copy_(VS)
        VA, VS = hva, hvs
    else:
        VA, VS = VA.to(DEV), VS.to(DEV)
    Pt = dev(rnd(synth.haar_orthogonal(m, rng, k).T).astype(np.float32), tdt)
    desc = E.layer_desc(plan, T, k, VA, VS, Pt, lengths=lengths)
    return plan, desc, (VA, VS, Pt)


@pytest.mark.parametrize("n,chunk,host_bases", [(5, 2, (True, False, True)), (1, 0, (True,)),
                                                (4, 0, (False, True)), (3, 1, (True, True, True))])
def test_several_modules_host_call_matches_device_inputs(n, chunk, host_bases):
    """eogp_compress_layers_host (the modules of a stack in one call, staging sets
    alternating between modules so that one module's copies overlap the previous
    one's compute) gives each module the results of eogp_compress_layer on the
    same inputs in device memory, bit for bit: modules of different shapes
    (different staging sizes in one workspace), host and device eigenbases,
    ragged chunks, per-example lengths, codes written into strided views of one
    output like a stack's, and the coordinates mode."""
    rng = np.random.default_rng(100 * n + chunk)
    T, B, k, m = 64, 5, 256, 2048
    shapes = [(768, 2304), (768, 768), (2304, 768)]
    lv = rng.integers(1, T + 1, B).astype(np.int32)
    lv[0] = T
    lengths = dev(lv)
    types = [_host_module(rng, di, do, T, m, k, host_bases[t % len(host_bases)], lengths)
             for t, (di, do) in enumerate(shapes)]
    descs, ah, sh, ad, sd = [], [], [], [], []
    for u in range(n):
        plan, desc, _ = types[u % len(types)]
        di, do = shapes[u % len(types)]
        a = torch.from_numpy(synth.round_to(rng.standard_normal((B, T, di)), "bf16").astype(np.float32))
        s = torch.from_numpy(synth.round_to(rng.standard_normal((B, T, do)) * 0.1, "bf16").astype(np.float32))
        a, s = a.to(torch.bfloat16), s.to(torch.bfloat16)
        ha, hs = E.host_empty(a.shape, torch.bfloat16), E.host_empty(s.shape, torch.bfloat16)
        ha.copy_(a)
        hs.copy_(s)
        descs.append(desc)
        ah.append(ha)
        sh.append(hs)
        ad.append(a.to(DEV))
        sd.append(s.to(DEV))
    wd = (k + 31) // 32
    codes = torch.zeros((B, n * wd), dtype=torch.int32, device=DEV)
    scales = torch.zeros((B, n), dtype=torch.float32, device=DEV)
    E.compress_layers_host(descs, ah, sh, E.OUT_CODES, DEV, chunk=chunk,
                           codes=[codes[:, u * wd:(u + 1) * wd] for u in range(n)],
                           scales=[scales[:, u] for u in range(n)])
    outs = E.compress_layers_host(descs, ah, sh, E.OUT_COORDS, DEV, chunk=chunk)
    if n == 1:
        assert E.compress_layers_host_workspace_size(descs, B, E.OUT_CODES, chunk) == \
            E.compress_host_workspace_size(descs[0], B, E.OUT_CODES, chunk)
    torch.cuda.synchronize()
    for u in range(n):
        c1, s1 = E.compress_layer(descs[u], ad[u], sd[u], E.OUT_CODES)
        x1 = E.compress_layer(descs[u], ad[u], sd[u], E.OUT_COORDS)
        torch.cuda.synchronize()
        assert torch.equal(codes[:, u * wd:(u + 1) * wd], c1), u
        assert torch.equal(scales[:, u], s1), u
        assert torch.equal(outs[u], x1), u
    E.sync_status()


def test_host_empty_memory_round_trip():
    """eogp_host_alloc memory (through host_empty): zero-filled, writable, copies
    to and from the device asynchronously, and is released with the tensor."""
    import gc
    t = E.host_empty((3, 1000, 7), torch.bfloat16)
    assert t.shape == (3, 1000, 7) and t.dtype == torch.bfloat16 and not t.is_cuda
    assert int(t.abs().sum()) == 0
    src = torch.randn(3, 1000, 7).to(torch.bfloat16)
    t.copy_(src)
    d = torch.empty_like(t, device=DEV)
    d.copy_(t, non_blocking=True)
    back = E.host_empty(t.shape, torch.bfloat16)
    back.copy_(d, non_blocking=True)
    torch.cuda.synchronize()
    assert torch.equal(back, src)
    del t, back
    gc.collect()


def test_host_alloc_size_classes():
    """eogp_host_alloc in each size class (base pages below 1 MB, blocks of a
    shared huge-page arena up to half a huge page, whole huge pages above):
    blocks are 4 KB aligned, never overlap while live, come back zero-filled
    after a freed block is reused, and copy to the device and back."""
    import ctypes
    L = E.lib()
    sizes = [64 << 10, 1 << 20, (3 << 20) + 123, 5 << 20, 17 << 20]
    ptrs = []
    for n in sizes:
        p = ctypes.c_void_p()
        assert L.eogp_host_alloc(n, ctypes.byref(p)) == E.OK
        assert p.value % 4096 == 0
        ctypes.memset(p.value, 0x5A, n)
        ptrs.append((p.value, n))
    spans = sorted(ptrs)
    for (a, na), (b, _) in zip(spans, spans[1:]):
        assert a + na <= b, "live blocks overlap"
    # free the middle blocks and take them again: the new blocks are zero-filled
    for p, n in ptrs[1:3]:
        assert L.eogp_host_free(ctypes.c_void_p(p)) == E.OK
    again = []
    for n in sizes[1:3]:
        p = ctypes.c_void_p()
        assert L.eogp_host_alloc(n, ctypes.byref(p)) == E.OK
        buf = (ctypes.c_uint8 * n).from_address(p.value)
        assert not any(bytes(buf)), "reused block not zero-filled"
        again.append((p.value, n))
    # device round trip through the largest arena-class block
    p, n = again[1]
    host = torch.frombuffer((ctypes.c_uint8 * n).from_address(p), dtype=torch.uint8)
    host.copy_(torch.randint(0, 256, (n,), dtype=torch.uint8))
    d = host.to(DEV, non_blocking=True)
    back = torch.empty_like(host).pin_memory()
    back.copy_(d, non_blocking=True)
    torch.cuda.synchronize()
    assert torch.equal(back, host)
    del host
    for p, _ in [ptrs[0], ptrs[3], ptrs[4]] + again:
        assert L.eogp_host_free(ctypes.c_void_p(p)) == E.OK


def test_bounded_wait_times_out_and_context_survives():
    """A kernel wait made to run out (an mbarrier nothing arrives on, a limit of
    2e6 cycles) reports EOGP_ETIMEOUT through eogp_sync_status, the report clears
    the status word, and the next library call on the same context succeeds."""
    assert E.selftest_wait_timeout(2_000_000) == E.ETIMEOUT
    assert E.lib().eogp_sync_status(None) == E.OK
    x = torch.randn(64, 256, device=DEV)
    codes, scales = torch.empty(64, 8, dtype=torch.int32, device=DEV), torch.empty(64, device=DEV)
    E.pack_sign(x, codes, scales)
    E.sync_status()
    bits, sc = O.onebit(x.cpu().double().numpy())
    assert np.array_equal(O.unpack_bits(codes.cpu().numpy().view(np.uint32), 256), bits)


def test_measure_peaks_rates():
    """eogp_measure_peaks: the e4m3 and e2m1 one-bit MMA rates and the popcount
    rate are finite and positive, the e2m1 MMA (K = 64 per instruction) outruns
    the e4m3 one (K = 32), and the probes leave no device error behind."""
    import math
    f8, f4, pc = E.measure_peaks()
    E.sync_status()
    for v in (f8, f4, pc):
        assert math.isfinite(v) and v > 0
    assert f4 > f8
