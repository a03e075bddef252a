"""eogp_compress_layer_static: compression for callers that cannot allocate.

Some callers cannot hand the library a workspace: a plugin whose host
framework owns every device allocation, a service held to a memory budget
fixed at start-up, a C program without an allocator. For them the library
offers eogp_compress_layer_static, which runs the normal compression kernels
on a scratch array built into the library. This test calls it through the C
ABI twice in a row and checks both results against eogp_compress_layer with a
caller workspace, then checks that an oversized batch is refused.
"""
import ctypes
import os
import re

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2609_37842_gb300 import eogp as E  # noqa: E402
from paper_2609_37842_gb300 import synth  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _static_bytes():
    """EOGP_STATIC_WORKSPACE_BYTES as the public header defines it."""
    with open(os.path.join(ROOT, "include", "eogp.h")) as f:
        m = re.search(r"#define\s+EOGP_STATIC_WORKSPACE_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", f.read())
    assert m, "EOGP_STATIC_WORKSPACE_BYTES not found in include/eogp.h"
    return int(m.group(1)) << int(m.group(2))


STATIC_BYTES = _static_bytes()


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_37842_gb300 import build
    build.build()
    E.lib()
    yield


def _module(dev):
    rng = np.random.default_rng(2024)
    d_in, d_out, T, m, k = 256, 384, 128, 1024, 256
    QA = synth.round_bf16(synth.haar_orthogonal(d_in, rng))
    QS = synth.round_bf16(synth.haar_orthogonal(d_out, rng))
    Pt = np.ascontiguousarray(synth.round_bf16(synth.haar_orthogonal(m, rng, k).T))
    plan = E.Plan.from_factors(synth.power_spectrum(d_out, 1.2), synth.power_spectrum(d_in, 1.2),
                               m, 0.1)
    bf = torch.bfloat16
    VA = plan.gather_rows(0, torch.from_numpy(np.ascontiguousarray(QA.T)).to(dev, bf))
    VS = plan.gather_rows(1, torch.from_numpy(np.ascontiguousarray(QS.T)).to(dev, bf))
    desc = E.layer_desc(plan, T, k, VA, VS, torch.from_numpy(Pt).to(dev, bf))
    return desc, rng, T, d_in, d_out, k


def _static_call(desc, a, s, mode, out=None, codes=None, scales=None):
    L = E.lib()
    stream = torch.cuda.current_stream().cuda_stream
    rc = L.eogp_compress_layer_static(
        ctypes.byref(desc), a.data_ptr(), s.data_ptr(), a.shape[0], mode,
        out.data_ptr() if out is not None else None, out.stride(0) if out is not None else 0,
        codes.data_ptr() if codes is not None else None, codes.stride(0) if codes is not None else 0,
        scales.data_ptr() if scales is not None else None, 1 if scales is not None else 0, stream)
    return rc


def test_static_scratch_matches_workspace_path():
    dev = torch.device("cuda:0")
    desc, rng, T, d_in, d_out, k = _module(dev)
    B = 6
    bf = torch.bfloat16
    a = torch.from_numpy(synth.round_bf16(rng.standard_normal((B, T, d_in)))).to(dev, bf)
    s = torch.from_numpy(synth.round_bf16(rng.standard_normal((B, T, d_out)) * 0.1)).to(dev, bf)
    assert E.compress_workspace_size(desc, B, E.OUT_CODES) <= STATIC_BYTES

    # Reference: the existing entry point with a caller-allocated workspace.
    codes_ref, scales_ref = E.compress_layer(desc, a, s, E.OUT_CODES)
    x_ref = E.compress_layer(desc, a, s, E.OUT_COORDS)
    E.sync_status()

    W = (k + 31) // 32
    for _ in range(2):  # two calls in a row share (and reuse) the built-in scratch
        codes = torch.full((B, W), -1, dtype=torch.int32, device=dev)
        scales = torch.full((B,), -1.0, dtype=torch.float32, device=dev)
        x = torch.full((B, k), float("nan"), dtype=torch.float32, device=dev)
        assert _static_call(desc, a, s, E.OUT_CODES, codes=codes, scales=scales) == E.OK, \
            E.lib().eogp_last_error()
        assert _static_call(desc, a, s, E.OUT_COORDS, out=x) == E.OK, E.lib().eogp_last_error()
        E.sync_status()
        assert torch.equal(codes, codes_ref)
        np.testing.assert_allclose(scales.cpu().numpy(), scales_ref.cpu().numpy(), rtol=1e-5)
        xr = x_ref.cpu().numpy().astype(np.float64)
        rel = np.linalg.norm(x.cpu().numpy() - xr, axis=1) / np.linalg.norm(xr, axis=1)
        assert rel.max() <= 2e-3


def test_static_scratch_rejects_oversized_batch():
    dev = torch.device("cuda:0")
    desc, rng, T, d_in, d_out, k = _module(dev)
    B = 256
    assert E.compress_workspace_size(desc, B, E.OUT_CODES) > STATIC_BYTES
    a = torch.zeros((B, T, d_in), dtype=torch.bfloat16, device=dev)
    s = torch.zeros((B, T, d_out), dtype=torch.bfloat16, device=dev)
    codes = torch.empty((B, (k + 31) // 32), dtype=torch.int32, device=dev)
    scales = torch.empty((B,), dtype=torch.float32, device=dev)
    assert _static_call(desc, a, s, E.OUT_CODES, codes=codes, scales=scales) == E.EUNSUPPORTED
    assert b"built-in scratch" in E.lib().eogp_last_error()
