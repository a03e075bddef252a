"""Python binding of libeogp (include/eogp.h): argument marshalling only.

Every computation runs in the library's CUDA kernels; PyTorch supplies device
memory and streams. Functions keep the C names without the ``eogp_`` prefix.
If libeogp.so has not been built, the first call raises: there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int, c_int32, c_size_t, c_uint32, c_void_p
from typing import Optional, Sequence, Tuple

import numpy as np

from . import build as _build

OK, EINVAL, EUNSUPPORTED, ECUDA, ETIMEOUT, EWORKSPACE, EDEVICE = 0, -1, -2, -3, -4, -5, -6
F32, BF16 = 0, 1
OUT_FIRST_STAGE, OUT_COORDS, OUT_CODES = 0, 1, 2
SCORE_CODES, SCORE_PAPER, SCORE_FP = 0, 1, 2
TOPK_MAX = 256
SRHT_MAX_M = 32768
K_ROTATE, K_CONTRACT, K_PROJECT, K_PACK, K_SCORE, K_SIMT = range(6)
KERNEL_KINDS = {K_ROTATE: "rotate", K_CONTRACT: "contract", K_PROJECT: "project", K_PACK: "pack",
                K_SCORE: "score", K_SIMT: "simt_f32"}

_ERRNAMES = {EINVAL: "EINVAL", EUNSUPPORTED: "EUNSUPPORTED", ECUDA: "ECUDA",
             ETIMEOUT: "ETIMEOUT", EWORKSPACE: "EWORKSPACE", EDEVICE: "EDEVICE"}


class EOGPError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{_ERRNAMES.get(code, code)}: {msg}")
        self.code = code


class PlanInfo(ctypes.Structure):
    _fields_ = [("d_in", c_int), ("d_out", c_int), ("m", c_int), ("nR", c_int), ("nC", c_int),
                ("n_tiles", c_int), ("lam", c_double)]


class LayerDesc(ctypes.Structure):
    _fields_ = [("d_in", c_int), ("d_out", c_int), ("T", c_int), ("m", c_int), ("k", c_int),
                ("dtype", c_int), ("VA", c_void_p), ("VS", c_void_p), ("Pt", c_void_p),
                ("plan", c_void_p), ("srht_signs", c_void_p), ("srht_rows", c_void_p),
                ("bias_A", c_void_p), ("lengths", c_void_p), ("bases_on_host", c_int)]


class EkfacDesc(ctypes.Structure):
    _fields_ = [("d_in", c_int), ("d_out", c_int), ("T", c_int), ("dtype", c_int),
                ("VA", c_void_p), ("VS", c_void_p)]


EXPORTS = {
    # name: (restype, argtypes)
    "eogp_last_error": (ctypes.c_char_p, []),
    "eogp_version": (ctypes.c_char_p, []),
    "eogp_sync_status": (c_int, [c_void_p]),
    "eogp_measure_peaks": (c_int, [POINTER(c_double), POINTER(c_double), POINTER(c_double)]),
    "eogp_selftest_wait_timeout": (c_int, [ctypes.c_longlong]),
    "eogp_profile_enable": (c_int, [c_int]),
    "eogp_set_option": (c_int, [c_int, c_int]),
    "eogp_get_option": (c_int, [c_int, POINTER(c_int)]),
    "eogp_profile_read": (c_int, [c_int, POINTER(c_int), POINTER(c_double), c_int]),
    "eogp_plan_layer": (c_int, [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_double,
                                POINTER(c_void_p)]),
    "eogp_plan_destroy": (None, [c_void_p]),
    "eogp_plan_get_info": (c_int, [c_void_p, POINTER(PlanInfo)]),
    "eogp_plan_get_retained": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
    "eogp_plan_get_sets": (c_int, [c_void_p, c_void_p, c_void_p]),
    "eogp_plan_gather_rows": (c_int, [c_void_p, c_int, c_int, c_void_p, c_int, c_void_p, c_void_p]),
    "eogp_compress_workspace_size": (c_int, [POINTER(LayerDesc), c_int, c_int, POINTER(c_size_t)]),
    "eogp_compress_layer": (c_int, [POINTER(LayerDesc), c_void_p, c_void_p, c_int, c_int, c_void_p,
                                    c_int, c_void_p, c_int, c_void_p, c_int, c_void_p, c_size_t,
                                    c_void_p]),
    "eogp_compress_layer_static": (c_int, [POINTER(LayerDesc), c_void_p, c_void_p, c_int, c_int,
                                           c_void_p, c_int, c_void_p, c_int, c_void_p, c_int,
                                           c_void_p]),
    "eogp_host_alloc": (c_int, [c_size_t, POINTER(c_void_p)]),
    "eogp_host_free": (c_int, [c_void_p]),
    "eogp_compress_host_workspace_size": (c_int, [POINTER(LayerDesc), c_int, c_int, c_int,
                                                  POINTER(c_size_t)]),
    "eogp_compress_layer_host": (c_int, [POINTER(LayerDesc), c_void_p, c_void_p, c_int, c_int, c_int,
                                         c_void_p, c_int, c_void_p, c_int, c_void_p, c_int, c_void_p,
                                         c_size_t, c_void_p]),
    "eogp_compress_layers_host_workspace_size": (c_int, [POINTER(POINTER(LayerDesc)), c_int, c_int, c_int, c_int,
                                                         POINTER(c_size_t)]),
    "eogp_compress_layers_host": (c_int, [POINTER(POINTER(LayerDesc)), c_int, POINTER(c_void_p), POINTER(c_void_p),
                                          c_int, c_int, c_int, POINTER(c_void_p), c_int, POINTER(c_void_p), c_int,
                                          POINTER(c_void_p), c_int, c_void_p, c_size_t, c_void_p]),
    "eogp_ekfac_workspace_size": (c_int, [POINTER(EkfacDesc), c_int, POINTER(c_size_t)]),
    "eogp_ekfac_accumulate": (c_int, [POINTER(EkfacDesc), c_void_p, c_void_p, c_int, c_void_p, c_int,
                                      c_int, c_void_p, c_size_t, c_void_p]),
    "eogp_fit_pca_workspace_size": (c_int, [c_int, c_int, c_int, POINTER(c_size_t)]),
    "eogp_fit_pca": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_void_p, c_int, c_int,
                             c_void_p, c_void_p, c_size_t, c_void_p]),
    "eogp_payload_bytes": (c_int, [c_void_p, c_int, POINTER(c_size_t)]),
    "eogp_payload_pack": (c_int, [c_void_p, c_int, c_void_p, c_int, c_int, c_void_p, c_int, c_void_p,
                                  c_size_t, c_void_p]),
    "eogp_payload_unpack": (c_int, [c_void_p, c_size_t, c_int, c_void_p, c_int, c_void_p, c_int,
                                    c_void_p, c_int, c_void_p]),
    "eogp_srht": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_void_p, c_int, c_void_p, c_int,
                          c_void_p, c_int, c_void_p, c_int, c_void_p]),
    "eogp_second_moment": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_int, c_int, c_void_p]),
    "eogp_fit_pca_from_moment_workspace_size": (c_int, [c_int, c_int, POINTER(c_size_t)]),
    "eogp_fit_pca_from_moment": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_void_p, c_int, c_int,
                                         c_void_p, c_void_p, c_size_t, c_void_p]),
    "eogp_pack_sign": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_int, c_void_p, c_int,
                               c_void_p]),
    "eogp_score_workspace_size": (c_int, [c_int, c_void_p, c_int, c_int, c_int, POINTER(c_size_t)]),
    "eogp_score": (c_int, [c_void_p, c_int, c_void_p, c_int, c_int, c_void_p, c_int, c_int,
                           c_void_p, c_int, c_void_p, c_int, c_int, c_void_p, c_int, c_void_p,
                           c_size_t, c_void_p]),
    "eogp_score_topk_workspace_size": (c_int, [c_int, c_void_p, c_int, c_int, c_int, c_int,
                                               POINTER(c_size_t)]),
    "eogp_score_topk": (c_int, [c_void_p, c_int, c_void_p, c_int, c_int, c_void_p, c_int, c_int,
                                c_void_p, c_int, c_void_p, c_int, c_int, c_int, c_void_p, c_int,
                                c_void_p, c_int, c_void_p, c_size_t, c_void_p]),
}

_LIB = None


def lib() -> ctypes.CDLL:
    """Load libeogp.so (built in-tree by build.py). Raises if it is missing."""
    global _LIB
    if _LIB is None:
        path = os.environ.get("EOGP_LIB") or _build.LIB   # EOGP_LIB: an alternative build
        if not os.path.exists(path):
            raise RuntimeError(f"libeogp.so is not built ({path}); run "
                               "`python -m paper_2609_37842_gb300.build` first")
        L = ctypes.CDLL(path)
        for name, (res, args) in EXPORTS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = L
    return _LIB


def _check(rc: int):
    if rc != OK:
        raise EOGPError(rc, lib().eogp_last_error().decode(errors="replace"))


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr()


def _rows(t, name: str):
    """Require a row-major matrix view (unit inner stride); returns t."""
    if t is not None and t.dim() >= 1 and t.numel() > 0 and t.stride(-1) != 1:
        raise ValueError(f"{name} must have unit stride along its last dimension")
    return t


def _dense(t, name: str):
    if t is not None and t.numel() > 0 and not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _stream(stream) -> Optional[int]:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def version() -> str:
    return lib().eogp_version().decode()


def sync_status(stream=None) -> None:
    _check(lib().eogp_sync_status(_stream(stream)))


def profile_enable(on: bool) -> None:
    _check(lib().eogp_profile_enable(1 if on else 0))


def profile_read(kind: int, reset: bool = True) -> Tuple[int, float]:
    """(launches, total device ms) of one kernel kind since the last reset."""
    n = c_int()
    ms = c_double()
    _check(lib().eogp_profile_read(int(kind), ctypes.byref(n), ctypes.byref(ms), 1 if reset else 0))
    return n.value, ms.value


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise ValueError(f"unsupported dtype {t.dtype}")


# ------------------------------------------------------------------- plan
class Plan:
    """Retained-set plan of one module (wraps eogp_plan*)."""

    def __init__(self, handle: int):
        self._h = c_void_p(handle)

    @classmethod
    def from_factors(cls, lam_S, lam_A, m: int, damping_rel: float) -> "Plan":
        lam_S = np.ascontiguousarray(lam_S, np.float64)
        lam_A = np.ascontiguousarray(lam_A, np.float64)
        h = c_void_p()
        _check(lib().eogp_plan_layer(lam_S.ctypes.data, lam_A.ctypes.data, None, len(lam_A),
                                     len(lam_S), int(m), float(damping_rel), ctypes.byref(h)))
        return cls(h.value)

    @classmethod
    def from_table(cls, Lambda, m: int, damping_rel: float) -> "Plan":
        Lam = np.ascontiguousarray(Lambda, np.float64)
        d_out, d_in = Lam.shape
        h = c_void_p()
        _check(lib().eogp_plan_layer(None, None, Lam.ctypes.data, d_in, d_out, int(m),
                                     float(damping_rel), ctypes.byref(h)))
        return cls(h.value)

    @property
    def handle(self) -> int:
        return self._h.value

    def info(self) -> PlanInfo:
        inf = PlanInfo()
        _check(lib().eogp_plan_get_info(self._h, ctypes.byref(inf)))
        return inf

    def retained(self) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
        m = self.info().m
        j = np.empty(m, np.int32)
        i = np.empty(m, np.int32)
        sc = np.empty(m, np.float32)
        _check(lib().eogp_plan_get_retained(self._h, j.ctypes.data, i.ctypes.data, sc.ctypes.data))
        return j, i, sc

    def sets(self) -> Tuple[np.ndarray, np.ndarray]:
        inf = self.info()
        R = np.empty(inf.nR, np.int32)
        C = np.empty(inf.nC, np.int32)
        _check(lib().eogp_plan_get_sets(self._h, R.ctypes.data, C.ctypes.data))
        return R, C

    def gather_rows(self, which: int, V_full, out=None, stream=None):
        """Retained eigenvector rows: which=0 -> V_A[C] [nC, d_in], 1 -> V_S[R] [nR, d_out]."""
        import torch
        inf = self.info()
        n = inf.nC if which == 0 else inf.nR
        d = inf.d_in if which == 0 else inf.d_out
        if out is None:
            out = torch.empty((n, d), dtype=V_full.dtype, device=V_full.device)
        _check(lib().eogp_plan_gather_rows(self._h, which, _dtype_code(V_full), _ptr(V_full),
                                           V_full.stride(0), _ptr(out), _stream(stream)))
        return out

    def __del__(self):
        if getattr(self, "_h", None) is not None and self._h.value and _LIB is not None:
            _LIB.eogp_plan_destroy(self._h)
            self._h = c_void_p()


# ------------------------------------------------------------- compression
def layer_desc(plan: Plan, T: int, k: int, VA, VS, Pt=None, srht_signs=None,
               srht_rows=None, bias_A=None, lengths=None) -> LayerDesc:
    """Descriptor of one module. It keeps references to the plan and tensors so
    their device memory outlives the descriptor. With Pt None and srht_rows
    given (int32 [k]; srht_signs int8 [m]), the second stage is the SRHT.
    bias_A (fp32 [nC]): the module's bias as a constant-1 input channel (the
    plan is over d_in + 1 inputs; VA [nC, d_in]). lengths (int32 [B]): tokens
    kept per example for the calls that use this descriptor. VA and VS may be
    host tensors (pinned): each call then copies them to its workspace."""
    inf = plan.info()
    _dense(VA, "VA")
    _dense(VS, "VS")
    _dense(Pt, "Pt")
    d_in = inf.d_in - (1 if bias_A is not None else 0)
    on_host = not VA.is_cuda
    if on_host != (not VS.is_cuda):
        raise ValueError("VA and VS must both be on the device or both in host memory")
    d = LayerDesc(d_in, inf.d_out, int(T), inf.m, int(k), _dtype_code(VA), _ptr(VA),
                  _ptr(VS), _ptr(Pt), plan.handle, _ptr(srht_signs), _ptr(srht_rows),
                  _ptr(bias_A), _ptr(lengths), 1 if on_host else 0)
    d._refs = (plan, VA, VS, Pt, srht_signs, srht_rows, bias_A, lengths)
    return d


def compress_workspace_size(desc: LayerDesc, B: int, out_mode: int) -> int:
    n = c_size_t()
    _check(lib().eogp_compress_workspace_size(ctypes.byref(desc), int(B), int(out_mode),
                                              ctypes.byref(n)))
    return n.value


def workspace(nbytes: int, device):
    import torch
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def compress_layer(desc: LayerDesc, a, s, out_mode: int, out=None, codes=None, scales=None,
                   ws=None, stream=None):
    """eogp_compress_layer on a [B, T, d_in], s [B, T, d_out]. Returns `out` (z or x) for
    FIRST_STAGE / COORDS, (codes, scales) for CODES. Output tensors may be given
    (strided rows: codes/scales of one module inside a wider store row)."""
    import torch
    _dense(a, "a")
    _dense(s, "s")
    _rows(out, "out")
    _rows(codes, "codes")
    B = a.shape[0]
    dev = a.device
    if ws is None:
        ws = workspace(compress_workspace_size(desc, B, out_mode), dev)
    if out_mode == OUT_CODES:
        if codes is None:
            codes = torch.empty((B, (desc.k + 31) // 32), dtype=torch.int32, device=dev)
        if scales is None:
            scales = torch.empty((B,), dtype=torch.float32, device=dev)
        ld_sc = scales.stride(0)
        _check(lib().eogp_compress_layer(ctypes.byref(desc), _ptr(a), _ptr(s), B, out_mode, None, 0,
                                         _ptr(codes), codes.stride(0), _ptr(scales), ld_sc,
                                         _ptr(ws), ws.numel(), _stream(stream)))
        return codes, scales
    width = desc.m if out_mode == OUT_FIRST_STAGE else desc.k
    if out is None:
        out = torch.empty((B, width), dtype=torch.float32, device=dev)
    _check(lib().eogp_compress_layer(ctypes.byref(desc), _ptr(a), _ptr(s), B, out_mode, _ptr(out),
                                     out.stride(0), None, 0, None, 0, _ptr(ws), ws.numel(),
                                     _stream(stream)))
    return out


def host_empty(shape, dtype):
    """A CPU tensor of `shape` / `dtype` in eogp_host_alloc memory (page-locked,
    huge-page backed, zero-filled); the memory is released with the tensor."""
    import numpy as np
    import torch
    import weakref
    nel = 1
    for d in shape:
        nel *= int(d)
    esz = torch.empty((), dtype=dtype).element_size()
    nbytes = max(1, nel * esz)
    p = c_void_p()
    _check(lib().eogp_host_alloc(nbytes, ctypes.byref(p)))
    buf = (ctypes.c_uint8 * nbytes).from_address(p.value)
    t = torch.from_numpy(np.frombuffer(buf, dtype=np.uint8)[:nel * esz]).view(dtype).view(*shape)
    weakref.finalize(buf, lib().eogp_host_free, p.value)
    t._eogp_host_buf = buf   # the finalizer runs once no tensor view holds the buffer
    return t


def compress_host_workspace_size(desc: LayerDesc, B: int, out_mode: int, chunk: int = 0) -> int:
    n = c_size_t()
    _check(lib().eogp_compress_host_workspace_size(ctypes.byref(desc), int(B), int(chunk),
                                                   int(out_mode), ctypes.byref(n)))
    return n.value


def compress_layer_host(desc: LayerDesc, a, s, out_mode: int, device, chunk: int = 0, out=None,
                        codes=None, scales=None, ws=None, stream=None):
    """eogp_compress_layer_host: a [B, T, d_in], s [B, T, d_out] in (page-locked)
    host memory, copied chunk by chunk by the call itself; outputs on `device`
    as for compress_layer."""
    import torch
    _dense(a, "a")
    _dense(s, "s")
    _rows(out, "out")
    _rows(codes, "codes")
    if a.is_cuda or s.is_cuda:
        raise ValueError("compress_layer_host takes host tensors (use compress_layer for device ones)")
    B = a.shape[0]
    if ws is None:
        ws = workspace(compress_host_workspace_size(desc, B, out_mode, chunk), device)
    if out_mode == OUT_CODES:
        if codes is None:
            codes = torch.empty((B, (desc.k + 31) // 32), dtype=torch.int32, device=device)
        if scales is None:
            scales = torch.empty((B,), dtype=torch.float32, device=device)
        _check(lib().eogp_compress_layer_host(ctypes.byref(desc), _ptr(a), _ptr(s), B, int(chunk),
                                              out_mode, None, 0, _ptr(codes), codes.stride(0),
                                              _ptr(scales), scales.stride(0), _ptr(ws), ws.numel(),
                                              _stream(stream)))
        return codes, scales
    width = desc.m if out_mode == OUT_FIRST_STAGE else desc.k
    if out is None:
        out = torch.empty((B, width), dtype=torch.float32, device=device)
    _check(lib().eogp_compress_layer_host(ctypes.byref(desc), _ptr(a), _ptr(s), B, int(chunk), out_mode,
                                          _ptr(out), out.stride(0), None, 0, None, 0, _ptr(ws),
                                          ws.numel(), _stream(stream)))
    return out


def _desc_array(descs):
    return (POINTER(LayerDesc) * len(descs))(*[ctypes.pointer(d) for d in descs])


def _ptr_array(ts):
    return (c_void_p * len(ts))(*[t.data_ptr() for t in ts])


def _common_ld(ts, name: str) -> int:
    lds = {t.stride(0) for t in ts}
    if len(lds) != 1:
        raise ValueError(f"{name}: every module's view must have the same leading dimension")
    return lds.pop()


def compress_layers_host_workspace_size(descs: Sequence[LayerDesc], B: int, out_mode: int, chunk: int = 0) -> int:
    n = c_size_t()
    _check(lib().eogp_compress_layers_host_workspace_size(_desc_array(descs), len(descs), int(B), int(chunk),
                                                          int(out_mode), ctypes.byref(n)))
    return n.value


def compress_layers_host(descs: Sequence[LayerDesc], a, s, out_mode: int, device, chunk: int = 0, out=None,
                         codes=None, scales=None, ws=None, stream=None):
    """eogp_compress_layers_host: module u compresses host tensors a[u] [B, T, d_in]
    and s[u] [B, T, d_out] (page-locked) into codes[u] / scales[u] (OUT_CODES) or
    out[u], all on `device`; the copies of one module overlap the compute of the
    previous one. Output views of one kind share one leading dimension."""
    import torch
    n = len(descs)
    if len(a) != n or len(s) != n:
        raise ValueError("one a and one s per descriptor")
    for t in list(a) + list(s):
        _dense(t, "a / s")
        if t.is_cuda:
            raise ValueError("compress_layers_host takes host tensors (use compress_layer for device ones)")
    B = a[0].shape[0]
    if any(t.shape[0] != B for t in list(a) + list(s)):
        raise ValueError("every module's a and s must hold the same B examples")
    if ws is None:
        ws = workspace(compress_layers_host_workspace_size(descs, B, out_mode, chunk), device)
    if out_mode == OUT_CODES:
        if codes is None:
            codes = [torch.empty((B, (d.k + 31) // 32), dtype=torch.int32, device=device) for d in descs]
        if scales is None:
            scales = [torch.empty((B,), dtype=torch.float32, device=device) for _ in descs]
        for t in codes:
            _rows(t, "codes")
        _check(lib().eogp_compress_layers_host(_desc_array(descs), n, _ptr_array(a), _ptr_array(s), B, int(chunk),
                                               out_mode, None, 0, _ptr_array(codes), _common_ld(codes, "codes"),
                                               _ptr_array(scales), _common_ld(scales, "scales"), _ptr(ws),
                                               ws.numel(), _stream(stream)))
        return codes, scales
    if out is None:
        out = [torch.empty((B, d.m if out_mode == OUT_FIRST_STAGE else d.k), dtype=torch.float32, device=device)
               for d in descs]
    for t in out:
        _rows(t, "out")
    _check(lib().eogp_compress_layers_host(_desc_array(descs), n, _ptr_array(a), _ptr_array(s), B, int(chunk),
                                           out_mode, _ptr_array(out), _common_ld(out, "out"), None, 0, None, 0,
                                           _ptr(ws), ws.numel(), _stream(stream)))
    return out


# ------------------------------------------------------------------ fit PCA
def ekfac_desc(T: int, VA, VS) -> EkfacDesc:
    """EK-FAC correction descriptor: VA [d_in, d_in], VS [d_out, d_out] with the
    eigenvectors as rows (full bases). Keeps references to the tensors."""
    _dense(VA, "VA")
    _dense(VS, "VS")
    d = EkfacDesc(VA.shape[1], VS.shape[1], int(T), _dtype_code(VA), _ptr(VA), _ptr(VS))
    d._refs = (VA, VS)
    return d


def ekfac_workspace_size(desc: EkfacDesc, B: int) -> int:
    n = c_size_t()
    _check(lib().eogp_ekfac_workspace_size(ctypes.byref(desc), int(B), ctypes.byref(n)))
    return n.value


def ekfac_accumulate(desc: EkfacDesc, a, s, sumsq=None, accumulate: bool = False, ws=None,
                     stream=None):
    """eogp_ekfac_accumulate: sumsq [d_out, d_in] fp64 (+)= sum_b (Q_S^T G_b Q_A)^2."""
    import torch
    _dense(a, "a")
    _dense(s, "s")
    B = a.shape[0]
    dev = a.device
    if sumsq is None:
        sumsq = torch.zeros((desc.d_out, desc.d_in), dtype=torch.float64, device=dev)
    _rows(sumsq, "sumsq")
    if ws is None:
        ws = workspace(ekfac_workspace_size(desc, B), dev)
    _check(lib().eogp_ekfac_accumulate(ctypes.byref(desc), _ptr(a), _ptr(s), B, _ptr(sumsq),
                                       sumsq.stride(0), 1 if accumulate else 0, _ptr(ws), ws.numel(),
                                       _stream(stream)))
    return sumsq


def fit_pca_workspace_size(n: int, m: int, k: int) -> int:
    v = c_size_t()
    _check(lib().eogp_fit_pca_workspace_size(int(n), int(m), int(k), ctypes.byref(v)))
    return v.value


def fit_pca(Z, k: int, pt_dtype: int = F32, ws=None, stream=None):
    """Top-k PCA directions of Z [n, m] (fp32, device): returns (Pt [k, m], eig [k])."""
    import torch
    _rows(Z, "Z")
    n, m = Z.shape
    if ws is None:
        ws = workspace(fit_pca_workspace_size(n, m, k), Z.device)
    Pt = torch.empty((k, m), dtype=torch.bfloat16 if pt_dtype == BF16 else torch.float32,
                     device=Z.device)
    eig = torch.empty((k,), dtype=torch.float32, device=Z.device)
    _check(lib().eogp_fit_pca(_ptr(Z), n, m, Z.stride(0), int(k), _ptr(Pt), Pt.stride(0), pt_dtype,
                              _ptr(eig), _ptr(ws), ws.numel(), _stream(stream)))
    return Pt, eig


# --------------------------------------------------------------- pack, score
def srht(z, signs, rows, x=None, codes=None, scales=None, want_x=True, want_codes=False,
         stream=None):
    """eogp_srht on z [B, m] fp32: returns x [B, k] and/or (codes, scales)."""
    import torch
    _rows(z, "z")
    B, m = z.shape
    k = rows.shape[0]
    if want_x and x is None:
        x = torch.empty((B, k), dtype=torch.float32, device=z.device)
    if want_codes:
        if codes is None:
            codes = torch.empty((B, (k + 31) // 32), dtype=torch.int32, device=z.device)
        if scales is None:
            scales = torch.empty((B,), dtype=torch.float32, device=z.device)
    _check(lib().eogp_srht(_ptr(z), B, m, z.stride(0), _ptr(signs), _ptr(rows), k,
                           _ptr(x) if want_x else None, x.stride(0) if want_x else 0,
                           _ptr(codes) if want_codes else None, codes.stride(0) if want_codes else 0,
                           _ptr(scales) if want_codes else None,
                           scales.stride(0) if want_codes else 0, _stream(stream)))
    if want_x and want_codes:
        return x, codes, scales
    return x if want_x else (codes, scales)


def pack_sign(x, codes=None, scales=None, stream=None):
    """Sign bits and ||x||_1/k of each row of x [B, k] (fp32, device)."""
    import torch
    _rows(x, "x")
    _rows(codes, "codes")
    B, k = x.shape
    if codes is None:
        codes = torch.empty((B, (k + 31) // 32), dtype=torch.int32, device=x.device)
    if scales is None:
        scales = torch.empty((B,), dtype=torch.float32, device=x.device)
    _check(lib().eogp_pack_sign(_ptr(x), B, k, x.stride(0), _ptr(codes), codes.stride(0),
                                _ptr(scales), scales.stride(0), _stream(stream)))
    return codes, scales


def score_workspace_size(N: int, ks: Sequence[int], mode: int, Q: int) -> int:
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    need = c_size_t()
    _check(lib().eogp_score_workspace_size(int(N), karr, len(ks), int(mode), int(Q), ctypes.byref(need)))
    return need.value


def score_topk_workspace_size(N: int, ks: Sequence[int], mode: int, Q: int, topk: int) -> int:
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    need = c_size_t()
    _check(lib().eogp_score_topk_workspace_size(int(N), karr, len(ks), int(mode), int(Q), int(topk),
                                                ctypes.byref(need)))
    return need.value


def score(train, train_scales, ks: Sequence[int], mode: int, query, query_scales=None, out=None,
          stream=None, ws=None):
    """eogp_score: returns scores [Q, N] fp32. A workspace of the size
    eogp_score_workspace_size asks for is allocated unless `ws` is given (pass an
    empty tensor to force the popcount kernels)."""
    import torch
    for t, nm in ((train, "train"), (query, "query"), (train_scales, "train_scales"),
                  (query_scales, "query_scales")):
        _rows(t, nm)
    N = train.shape[0]
    Q = query.shape[0]
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    if out is None:
        out = torch.empty((Q, N), dtype=torch.float32, device=train.device)
    ts_ld = train_scales.stride(0) if train_scales is not None else 0
    qs_ld = query_scales.stride(0) if query_scales is not None else 0
    if ws is None:
        need = c_size_t()
        _check(lib().eogp_score_workspace_size(N, karr, len(ks), int(mode), Q, ctypes.byref(need)))
        ws = workspace(need.value, train.device) if need.value else None
    _check(lib().eogp_score(_ptr(train), train.stride(0), _ptr(train_scales), ts_ld, N, karr,
                            len(ks), int(mode), _ptr(query), query.stride(0), _ptr(query_scales),
                            qs_ld, Q, _ptr(out), out.stride(0), _ptr(ws),
                            ws.numel() if ws is not None else 0, _stream(stream)))
    return out


def score_topk(train, train_scales, ks: Sequence[int], mode: int, query, topk: int,
               query_scales=None, ws=None, stream=None):
    """eogp_score_topk: per query the `topk` best stored rows. Returns
    (scores [Q, topk] fp32, index [Q, topk] int32), score descending, equal
    scores by lower row; (-inf, -1) past N."""
    import torch
    for t, nm in ((train, "train"), (query, "query"), (train_scales, "train_scales"),
                  (query_scales, "query_scales")):
        _rows(t, nm)
    N = train.shape[0]
    Q = query.shape[0]
    dev = query.device
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    top_s = torch.empty((Q, topk), dtype=torch.float32, device=dev)
    top_i = torch.empty((Q, topk), dtype=torch.int32, device=dev)
    if ws is None:
        need = c_size_t()
        _check(lib().eogp_score_topk_workspace_size(N, karr, len(ks), int(mode), Q, int(topk),
                                                    ctypes.byref(need)))
        ws = workspace(need.value, dev)
    ts_ld = train_scales.stride(0) if train_scales is not None else 0
    qs_ld = query_scales.stride(0) if query_scales is not None else 0
    _check(lib().eogp_score_topk(_ptr(train), train.stride(0), _ptr(train_scales), ts_ld, N, karr,
                                 len(ks), int(mode), _ptr(query), query.stride(0),
                                 _ptr(query_scales), qs_ld, Q, int(topk), _ptr(top_s),
                                 top_s.stride(0), _ptr(top_i), top_i.stride(0), _ptr(ws), ws.numel(),
                                 _stream(stream)))
    return top_s, top_i


def payload_bytes(ks: Sequence[int]) -> int:
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    n = c_size_t()
    _check(lib().eogp_payload_bytes(karr, len(ks), ctypes.byref(n)))
    return n.value


def payload_pack(codes, scales, ks: Sequence[int], out=None, stream=None):
    """Store records [N, payload_bytes(ks)] uint8 (device) from codes and scales."""
    import torch
    _rows(codes, "codes")
    _rows(scales, "scales")
    N = codes.shape[0]
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    if out is None:
        out = torch.empty((N, payload_bytes(ks)), dtype=torch.uint8, device=codes.device)
    sc = scales if scales.dim() == 2 else scales[:, None]
    _check(lib().eogp_payload_pack(_ptr(codes), codes.stride(0), _ptr(sc), sc.stride(0), N, karr, len(ks),
                                   _ptr(out), out.stride(0), _stream(stream)))
    return out


def payload_unpack(payload, ks: Sequence[int], stream=None):
    """(codes [N, W] int32, scales [N, U] fp32) from store records (device)."""
    import torch
    _rows(payload, "payload")
    N = payload.shape[0]
    karr = (c_int * len(ks))(*[int(k) for k in ks])
    W = sum((int(k) + 31) // 32 for k in ks)
    codes = torch.empty((N, W), dtype=torch.int32, device=payload.device)
    scales = torch.empty((N, len(ks)), dtype=torch.float32, device=payload.device)
    _check(lib().eogp_payload_unpack(_ptr(payload), payload.stride(0), N, karr, len(ks), _ptr(codes),
                                     codes.stride(0), _ptr(scales), scales.stride(0), _stream(stream)))
    return codes, scales


def write_store(path: str, payload) -> None:
    """Write store records (rows of payload_pack) to a file, back to back."""
    with open(path, "wb") as f:
        f.write(payload.cpu().numpy().tobytes())


def read_store(path: str, ks: Sequence[int], device) -> "torch.Tensor":
    """Read a file of store records back as a [N, payload_bytes(ks)] uint8 tensor."""
    import torch
    rb = payload_bytes(ks)
    raw = np.fromfile(path, dtype=np.uint8)
    if raw.size % rb:
        raise ValueError(f"{path}: {raw.size} bytes is not a whole number of {rb}-byte records")
    return torch.from_numpy(raw.reshape(-1, rb)).to(device)


OPT_SCORE_OPERAND = 0   # 0: e2m1 where it applies (default), 1: e4m3
OPT_TOPK_PATH = 1       # 0: by size (default), 1: fused ranking, 2: dense scores + ranking kernel


def set_option(option: int, value: int) -> None:
    """eogp_set_option: a process-wide dispatch choice between implementations
    with identical results (read by the workspace queries and the calls)."""
    _check(lib().eogp_set_option(option, value))


def get_option(option: int) -> int:
    v = c_int()
    _check(lib().eogp_get_option(option, ctypes.byref(v)))
    return v.value


class options:
    """Context manager setting dispatch options and restoring them on exit:
    `with options(score_operand=1, topk_path=2): ...`."""

    def __init__(self, score_operand: Optional[int] = None, topk_path: Optional[int] = None):
        self.want = {OPT_SCORE_OPERAND: score_operand, OPT_TOPK_PATH: topk_path}
        self.old = {}

    def __enter__(self):
        for o, v in self.want.items():
            if v is not None:
                self.old[o] = get_option(o)
                set_option(o, v)
        return self

    def __exit__(self, *exc):
        for o, v in self.old.items():
            set_option(o, v)
        return False


def measure_peaks() -> Tuple[float, float, float]:
    """(e4m3 and e2m1 tensor-core TFLOP/s, XOR + popcount words/s) measured on the
    current device."""
    f8 = c_double()
    f4 = c_double()
    pc = c_double()
    _check(lib().eogp_measure_peaks(ctypes.byref(f8), ctypes.byref(f4), ctypes.byref(pc)))
    return f8.value, f4.value, pc.value


def selftest_wait_timeout(limit_cycles: int = 2_000_000) -> int:
    """eogp_selftest_wait_timeout: status code of a wait made to run out (ETIMEOUT
    when the bounded-wait path works)."""
    return lib().eogp_selftest_wait_timeout(int(limit_cycles))


def second_moment(Z, C=None, accumulate: bool = False, stream=None):
    """eogp_second_moment: C [m, m] fp64 (+)= Z^T Z for Z [n, m] fp32 (device)."""
    import torch
    _rows(Z, "Z")
    n, m = Z.shape
    if C is None:
        C = torch.zeros((m, m), dtype=torch.float64, device=Z.device)
    _rows(C, "C")
    _check(lib().eogp_second_moment(_ptr(Z), n, m, Z.stride(0), _ptr(C), C.stride(0), 1 if accumulate else 0,
                                    _stream(stream)))
    return C


def fit_pca_from_moment(C, n_total: int, k: int, pt_dtype: int = F32, stream=None):
    """eogp_fit_pca_from_moment: (Pt [k, m], eig [k]) for the summed second moment C of n_total rows."""
    import torch
    _rows(C, "C")
    m = C.shape[0]
    need = c_size_t()
    _check(lib().eogp_fit_pca_from_moment_workspace_size(m, int(k), ctypes.byref(need)))
    ws = workspace(need.value, C.device)
    Pt = torch.empty((k, m), dtype=torch.float32 if pt_dtype == F32 else torch.bfloat16, device=C.device)
    eig = torch.empty((k,), dtype=torch.float32, device=C.device)
    _check(lib().eogp_fit_pca_from_moment(_ptr(C), m, C.stride(0), int(n_total), int(k), _ptr(Pt), Pt.stride(0),
                                          int(pt_dtype), _ptr(eig), _ptr(ws), ws.numel(), _stream(stream)))
    return Pt, eig
