"""CPU checks of the C ABI: the library loads, exports every function that
include/eogp.h declares, rejects bad arguments on the host, and its host-side
retained-set plan matches the oracle's selection exactly."""
import os
import re
import subprocess

import numpy as np
import pytest

from oracle import eogp_oracle as O
from paper_2609_37842_gb300 import build as B
from paper_2609_37842_gb300 import eogp as E
from paper_2609_37842_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    E.lib()


def declared_functions():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            txt = open(os.path.join(inc, f)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names |= set(re.findall(r"\b(eogp_\w+)\s*\(", txt))
    return sorted(names)


def test_every_declared_symbol_is_exported():
    names = declared_functions()
    assert len(names) >= 14
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (eogp_\w+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert n in E.EXPORTS, f"binding lacks {n}"
    # nothing but the ABI leaks out of the library
    assert all(n.startswith("eogp_") for n in exported)


def test_version_and_error_string():
    assert "sm_103a" in E.version()
    assert isinstance(E.lib().eogp_last_error(), bytes)


@pytest.mark.parametrize("d_in,d_out,m,alpha,rel", [
    (64, 64, 512, 1.5, 1e-3),      # the tiny fp32 workload: 6 ties at the boundary
    (8, 8, 7, 1.5, 0.1),           # cut inside a tie group
    (8, 8, 64, 1.0, 0.1),          # keep everything
    (768, 2304, 4096, 1.2, 0.1),   # GPT-2 c_attn
    (3072, 768, 4096, 1.2, 0.1),   # GPT-2 mlp c_proj
    (33, 17, 100, 0.7, 0.1),       # ragged sizes
])
def test_plan_matches_oracle_selection(d_in, d_out, m, alpha, rel):
    lamA = synth.power_spectrum(d_in, alpha)
    lamS = synth.power_spectrum(d_out, alpha)
    plan = E.Plan.from_factors(lamS, lamA, m, rel)
    j, i, sc = plan.retained()
    Lam = O.kfac_eigenvalues(lamS, lamA)
    jo, io = O.select_retained(Lam, m)
    np.testing.assert_array_equal(j, jo)
    np.testing.assert_array_equal(i, io)
    lam = O.damping(Lam, rel)
    inf = plan.info()
    assert inf.lam == pytest.approx(lam, rel=1e-12)
    want = (1.0 / np.sqrt(Lam[jo, io] + lam)).astype(np.float32)
    np.testing.assert_allclose(sc, want, rtol=2e-7, atol=0)
    R, C = plan.sets()
    np.testing.assert_array_equal(R, np.unique(jo))
    np.testing.assert_array_equal(C, np.unique(io))
    assert inf.nR == len(R) and inf.nC == len(C)


def test_plan_full_table_form():
    rng = np.random.default_rng(3)
    Lam = rng.uniform(0, 1, (20, 12))
    Lam[3, 4] = Lam[5, 6] = Lam[0, 0] = 0.99999   # ties in the table
    plan = E.Plan.from_table(Lam, 37, 0.1)
    j, i, _ = plan.retained()
    jo, io = O.select_retained(Lam, 37)
    np.testing.assert_array_equal(j, jo)
    np.testing.assert_array_equal(i, io)


@pytest.mark.parametrize("kwargs,code", [
    (dict(m=0), E.EINVAL), (dict(m=10_000), E.EINVAL), (dict(rel=-1.0), E.EINVAL),
    (dict(bad_lam=True), E.EINVAL)])
def test_plan_rejects_bad_arguments(kwargs, code):
    lam = np.arange(1, 9, dtype=np.float64) ** -1.0
    if kwargs.get("bad_lam"):
        lam = lam.copy()
        lam[2] = np.nan
    with pytest.raises(E.EOGPError) as ei:
        E.Plan.from_factors(lam, lam, kwargs.get("m", 10), kwargs.get("rel", 0.1))
    assert ei.value.code == code


def test_host_only_plan_is_rejected_by_compress():
    lam = np.arange(1, 9, dtype=np.float64) ** -1.0
    plan = E.Plan.from_factors(lam, lam, 10, 0.1)
    desc = E.LayerDesc(8, 8, 4, 10, 4, E.F32, 16, 16, 16, plan.handle)
    import ctypes
    n = ctypes.c_size_t()
    assert E.lib().eogp_compress_workspace_size(ctypes.byref(desc), 2, E.OUT_CODES, ctypes.byref(n)) == 0
    rc = E.lib().eogp_compress_layer(ctypes.byref(desc), 16, 16, 2, E.OUT_CODES, None, 0, 16, 1, 16,
                                     1, 256, n.value, None)
    assert rc == E.EINVAL


def test_host_argument_checks():
    L = E.lib()
    import ctypes
    n = ctypes.c_size_t()
    assert L.eogp_fit_pca_workspace_size(10, 20, 0, ctypes.byref(n)) == E.EINVAL
    assert L.eogp_fit_pca_workspace_size(10, 20, 11, ctypes.byref(n)) == E.EINVAL
    assert L.eogp_fit_pca_workspace_size(10, 20, 5, ctypes.byref(n)) == E.OK and n.value > 0
    assert L.eogp_pack_sign(None, -1, 8, 8, None, 1, None, 1, None) == E.EINVAL
    assert L.eogp_pack_sign(None, 4, 0, 8, None, 1, None, 1, None) == E.EINVAL
    assert L.eogp_pack_sign(None, 0, 8, 8, None, 1, None, 1, None) == E.OK   # empty batch
    ks = (ctypes.c_int * 2)(32, 0)
    assert L.eogp_score(16, 2, 16, 2, 4, ks, 2, 0, 16, 2, 16, 2, 4, 16, 4, None, 0, None) == E.EINVAL
    assert L.eogp_compress_workspace_size(None, 1, 0, ctypes.byref(n)) == E.EINVAL


def test_topk_host_argument_checks():
    L = E.lib()
    import ctypes
    n = ctypes.c_size_t()
    ks = (ctypes.c_int * 2)(1024, 1024)
    for bad_k in (0, E.TOPK_MAX + 1):
        assert L.eogp_score_topk_workspace_size(100, ks, 2, E.SCORE_CODES, 64, bad_k,
                                                ctypes.byref(n)) == E.EINVAL
    assert L.eogp_score_topk_workspace_size(100, ks, 2, E.SCORE_CODES, 64, 10, ctypes.byref(n)) == E.OK
    assert n.value > 0
    assert L.eogp_score_topk_workspace_size(100, ks, 2, E.SCORE_CODES, 0, 10, ctypes.byref(n)) == E.OK
    assert n.value == 0
    # bad mode, bad topk, missing outputs: rejected before any device work
    args = [16, 32, 16, 2, 100, ks, 2, 7, 16, 32, 16, 2, 64, 10, 16, 10, 16, 10, 256, 1 << 20, None]
    assert L.eogp_score_topk(*args) == E.EINVAL
    args[7] = E.SCORE_CODES
    args[13] = 0
    assert L.eogp_score_topk(*args) == E.EINVAL
    args[13] = 10
    args[14] = None
    assert L.eogp_score_topk(*args) == E.EINVAL
    args[14] = 16
    args[15] = 5     # ld_top_scores < topk
    assert L.eogp_score_topk(*args) == E.EINVAL
    args[15] = 10
    args[19] = 0     # workspace too small
    assert L.eogp_score_topk(*args) == E.EWORKSPACE


def test_host_input_call_argument_checks():
    """eogp_compress_layer_host / _workspace_size: argument checks that run before
    any device work (no GPU needed)."""
    import ctypes
    lam = np.arange(1, 9, dtype=np.float64) ** -1.0
    plan = E.Plan.from_factors(lam, lam, 10, 0.1)
    desc = E.LayerDesc(8, 8, 64, 10, 4, E.F32, 16, 16, 16, plan.handle)   # T = 64: 2 KB of a per example
    L = E.lib()
    n1, n2, n0 = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
    assert L.eogp_compress_host_workspace_size(ctypes.byref(desc), 6, 1, E.OUT_CODES, ctypes.byref(n1)) == E.OK
    assert L.eogp_compress_host_workspace_size(ctypes.byref(desc), 6, 2, E.OUT_CODES, ctypes.byref(n2)) == E.OK
    assert L.eogp_compress_host_workspace_size(ctypes.byref(desc), 6, 0, E.OUT_CODES, ctypes.byref(n0)) == E.OK
    assert 0 < n1.value < n2.value <= n0.value   # bigger chunks stage more; the default takes all 6
    assert L.eogp_compress_host_workspace_size(ctypes.byref(desc), 6, -1, E.OUT_CODES,
                                               ctypes.byref(n1)) == E.EINVAL
    assert L.eogp_compress_host_workspace_size(None, 6, 0, E.OUT_CODES, ctypes.byref(n1)) == E.EINVAL
    args = [ctypes.byref(desc), 16, 16, 2, 0, E.OUT_CODES, None, 0, 16, 1, 16, 1, 256, n0.value, None]
    assert L.eogp_compress_layer_host(*args) == E.EINVAL          # host-only plan
    args[4] = -1
    assert L.eogp_compress_layer_host(*args) == E.EINVAL          # negative chunk
    args[4], args[3] = 0, 0
    assert L.eogp_compress_layer_host(*args) == E.OK              # empty batch: nothing to do
    args[3], args[12] = 2, None
    assert L.eogp_compress_layer_host(*args) == E.EWORKSPACE


def test_several_modules_host_call_argument_checks():
    """eogp_compress_layers_host / _workspace_size: argument checks that run before
    any device work, and the workspace of one module equals the one-module call's."""
    import ctypes
    lam = np.arange(1, 9, dtype=np.float64) ** -1.0
    plan = E.Plan.from_factors(lam, lam, 10, 0.1)
    desc = E.LayerDesc(8, 8, 64, 10, 4, E.F32, 16, 16, 16, plan.handle)
    desc2 = E.LayerDesc(8, 8, 32, 10, 4, E.F32, 16, 16, 16, plan.handle)   # T = 32: smaller staging
    L = E.lib()
    one, two, ref = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
    arr1 = E._desc_array([desc])
    arr2 = E._desc_array([desc, desc2])
    assert L.eogp_compress_host_workspace_size(ctypes.byref(desc), 6, 2, E.OUT_CODES, ctypes.byref(ref)) == E.OK
    assert L.eogp_compress_layers_host_workspace_size(arr1, 1, 6, 2, E.OUT_CODES, ctypes.byref(one)) == E.OK
    assert one.value == ref.value
    assert L.eogp_compress_layers_host_workspace_size(arr2, 2, 6, 2, E.OUT_CODES, ctypes.byref(two)) == E.OK
    assert two.value > one.value    # two staging sets
    assert L.eogp_compress_layers_host_workspace_size(arr2, 0, 6, 2, E.OUT_CODES, ctypes.byref(two)) == E.EINVAL
    assert L.eogp_compress_layers_host_workspace_size(None, 1, 6, 2, E.OUT_CODES, ctypes.byref(two)) == E.EINVAL
    assert L.eogp_compress_layers_host_workspace_size(arr1, 1, 6, -1, E.OUT_CODES, ctypes.byref(two)) == E.EINVAL
    ptrs = (ctypes.c_void_p * 2)(16, 16)
    args = [arr2, 2, ptrs, ptrs, 2, 0, E.OUT_CODES, None, 0, ptrs, 16, ptrs, 1, 256, two.value, None]
    assert L.eogp_compress_layers_host(*args) == E.EINVAL          # host-only plan
    args[1] = 0
    assert L.eogp_compress_layers_host(*args) == E.EINVAL          # n < 1
    args[1], args[2] = 2, None
    assert L.eogp_compress_layers_host(*args) == E.EINVAL          # no a array
    args[2], args[9] = ptrs, None
    assert L.eogp_compress_layers_host(*args) == E.EINVAL          # no codes array
    args[9], args[4] = ptrs, 0
    assert L.eogp_compress_layers_host(*args) == E.OK              # empty batch: nothing to do
    args[4], args[13] = 2, None
    assert L.eogp_compress_layers_host(*args) == E.EWORKSPACE


def test_selftest_wait_argument_checks():
    """eogp_selftest_wait_timeout refuses limits outside [1, 1e9] before any device call."""
    L = E.lib()
    assert L.eogp_selftest_wait_timeout(0) == E.EINVAL
    assert L.eogp_selftest_wait_timeout(-5) == E.EINVAL
    assert L.eogp_selftest_wait_timeout(10 ** 10) == E.EINVAL


def test_host_alloc_argument_checks():
    """eogp_host_alloc / eogp_host_free: argument checks, and clean failure (or
    success, with a GPU present) of the registration."""
    import ctypes
    L = E.lib()
    p = ctypes.c_void_p()
    assert L.eogp_host_alloc(0, ctypes.byref(p)) == E.EINVAL and not p.value
    assert L.eogp_host_alloc(4096, None) == E.EINVAL
    assert L.eogp_host_free(None) == E.OK
    assert L.eogp_host_free(ctypes.c_void_p(4096)) == E.EINVAL   # not from eogp_host_alloc
    rc = L.eogp_host_alloc(4096, ctypes.byref(p))
    if rc == E.OK:          # a device is present: the region is usable and released
        ctypes.memset(p.value, 7, 4096)
        assert L.eogp_host_free(p) == E.OK
    else:                   # no device: registration fails and nothing is handed out
        assert rc == E.ECUDA and not p.value
