"""Seeded synthetic workloads for the EOGP hot path.

This module only draws random inputs and describes workload shapes. It holds
none of the method's arithmetic (no selection, scaling, projection, sign or
score step), so both the CUDA path and the CPU oracle can be fed from it
without sharing any computation.

The shapes follow the paper's evaluated models: GPT-2 small attention/MLP
linears at 512-token WikiText-2 blocks, and OLMo 2 1B / 7B / 32B linears at
up to 2048 tokens (App. C.1-C.2). No dataset or checkpoint is used: inputs are
Gaussian activations a_t and output gradients s_t, Haar-orthogonal Kronecker
eigenbases and power-law or per-channel eigenvalue spectra.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

# Role ids used to derive independent seed streams.
ROLE_A, ROLE_S, ROLE_QA, ROLE_QS, ROLE_QUERY_A, ROLE_QUERY_S, ROLE_FIT_A, ROLE_FIT_S, \
    ROLE_CODES, ROLE_SCALES, ROLE_P, ROLE_Z, ROLE_CHANNEL, ROLE_SRHT = range(14)


@dataclasses.dataclass(frozen=True)
class Module:
    name: str
    d_in: int
    d_out: int
    gelu_input: bool = False  # input activations pass through GELU (GPT-2 mlp c_proj)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    dtype: str                 # "f32" or "bf16": dtype of a, s, eigenbases and P
    modules: Tuple[Module, ...]
    T: int                     # tokens per example
    N: int                     # stored training examples
    m: int                     # retained first-stage coordinates per module
    k: int                     # PCA output coordinates (= sign bits) per module
    Q: int                     # queries
    spectrum: str              # "power" | "channel"
    alpha: float               # power-law exponent for "power" spectra
    damping_rel: float         # relative damping coefficient
    a_std: float = 1.0
    s_std: float = 1.0
    seed: int = 0
    fit_n: int = 0             # examples in the PCA fitting stream (0 = N)

    @property
    def n_modules(self) -> int:
        return len(self.modules)


def _gpt2_modules() -> Tuple[Module, ...]:
    mods = []
    for blk in range(12):
        mods += [Module(f"h{blk}.attn.c_attn", 768, 2304),
                 Module(f"h{blk}.attn.c_proj", 768, 768),
                 Module(f"h{blk}.mlp.c_fc", 768, 3072),
                 Module(f"h{blk}.mlp.c_proj", 3072, 768, gelu_input=True)]
    return tuple(mods)


def _olmo_modules(layers: int, d: int, ff: int) -> Tuple[Module, ...]:
    mods = []
    for l in range(layers):
        for nm in ("q_proj", "k_proj", "v_proj", "o_proj"):
            mods.append(Module(f"l{l}.attn.{nm}", d, d))
        mods += [Module(f"l{l}.mlp.gate_proj", d, ff), Module(f"l{l}.mlp.up_proj", d, ff),
                 Module(f"l{l}.mlp.down_proj", ff, d)]
    return tuple(mods)


WORKLOADS = {
    # Tiny single layer, fp32 everywhere.
    "tiny_f32": Workload("tiny_f32", "f32", (Module("layer", 64, 64),), T=16, N=256, m=512, k=128,
                         Q=8, spectrum="power", alpha=1.5, damping_rel=1e-3, seed=101),
    # GPT-2 small stack (48 linears), 512-token blocks.
    "gpt2_small_bf16": Workload("gpt2_small_bf16", "bf16", _gpt2_modules(), T=512, N=16384, m=4096,
                                k=1024, Q=1024, spectrum="power", alpha=1.2, damping_rel=0.1,
                                a_std=1.0, s_std=0.1, seed=202, fit_n=10000),
    # OLMo 2 1B stack (112 linears), 2048 tokens, per-channel log-uniform scales.
    "olmo2_1b_bf16": Workload("olmo2_1b_bf16", "bf16", _olmo_modules(16, 2048, 8192), T=2048,
                              N=65536, m=8192, k=2048, Q=4096, spectrum="channel", alpha=0.0,
                              damping_rel=0.1, seed=303, fit_n=10000),
    # OLMo 2 7B stack (224 linears), eigenbases streamed from host-pinned memory.
    "olmo2_7b_bf16": Workload("olmo2_7b_bf16", "bf16", _olmo_modules(32, 4096, 11008), T=2048,
                              N=32768, m=8192, k=2048, Q=1024, spectrum="power", alpha=1.0,
                              damping_rel=0.1, a_std=1.0, s_std=0.1, seed=404, fit_n=10000),
    # OLMo 2 32B gate projection, one layer.
    "olmo2_32b_gate_bf16": Workload("olmo2_32b_gate_bf16", "bf16",
                                    (Module("l0.mlp.gate_proj", 5120, 27648),), T=2048, N=4096,
                                    m=8192, k=2048, Q=0, spectrum="power", alpha=1.0,
                                    damping_rel=0.1, a_std=1.0, s_std=0.1, seed=505, fit_n=4096),
}

# Scoring-only sweep: stored one-bit codes with log-normal scales.
SCAN = dict(name="scan_16k", N=4_194_304, k=16384, Qs=(1, 64, 1024, 8192), seed=606,
            scale_sigma=0.5)


def rng_for(seed: int, role: int, *extra: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([seed, role, *extra]))


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even) directly from float64/float32.

    Returns float32 holding bf16-representable values. Rounding is done on the
    8-bit significand from frexp so a float64 input is rounded once.
    """
    x = np.asarray(x, dtype=np.float64)
    mant, ex = np.frexp(x)
    r = np.ldexp(np.rint(np.ldexp(mant, 8)), ex - 8)
    return r.astype(np.float32)


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return round_bf16(x)
    if dtype == "f32":
        return np.asarray(x, dtype=np.float64).astype(np.float32)
    raise ValueError(dtype)


def haar_orthogonal(d: int, rng: np.random.Generator, n_cols: Optional[int] = None) -> np.ndarray:
    """Haar-distributed orthogonal matrix (or its first n_cols columns) in float64:
    QR of a Gaussian matrix with column signs fixed by sign(diag R)."""
    n_cols = d if n_cols is None else n_cols
    g = rng.standard_normal((d, n_cols))
    q, r = np.linalg.qr(g)
    sgn = np.sign(np.diag(r))
    sgn[sgn == 0] = 1.0
    return q * sgn[None, :]


def power_spectrum(d: int, alpha: float) -> np.ndarray:
    """lambda_k = k^(-alpha), k = 1..d, float64, descending."""
    return np.arange(1, d + 1, dtype=np.float64) ** (-alpha)


def gelu_exact(x: np.ndarray) -> np.ndarray:
    from scipy.special import erf
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


@dataclasses.dataclass
class LayerSpec:
    """Per-module synthetic curvature: eigenbases and factor spectra.

    Q_A (d_in x d_in) and Q_S (d_out x d_out) hold eigenvectors as COLUMNS,
    sorted by eigenvalue descending, already rounded to the workload dtype.
    lam_A, lam_S are float64 descending spectra.
    """
    d_in: int
    d_out: int
    Q_A: np.ndarray
    Q_S: np.ndarray
    lam_A: np.ndarray
    lam_S: np.ndarray
    chan_A: Optional[np.ndarray] = None  # per-channel std of a ("channel" spectra)
    chan_S: Optional[np.ndarray] = None


def layer_spec(w: Workload, module_index: int, cols_A: Optional[int] = None,
               cols_S: Optional[int] = None) -> LayerSpec:
    """Eigenbases and spectra of one module.

    cols_A / cols_S keep only the leading eigenvectors (the rest are never
    read by the hot path); None keeps all of them.
    """
    mod = w.modules[module_index]
    if w.spectrum == "power":
        lam_A = power_spectrum(mod.d_in, w.alpha)
        lam_S = power_spectrum(mod.d_out, w.alpha)
        QA = haar_orthogonal(mod.d_in, rng_for(w.seed, ROLE_QA, module_index), cols_A)
        QS = haar_orthogonal(mod.d_out, rng_for(w.seed, ROLE_QS, module_index), cols_S)
        return LayerSpec(mod.d_in, mod.d_out, round_to(QA, w.dtype), round_to(QS, w.dtype),
                         lam_A, lam_S)
    if w.spectrum == "channel":
        r = rng_for(w.seed, ROLE_CHANNEL, module_index)
        sa = np.exp(r.uniform(math.log(0.1), math.log(10.0), mod.d_in))
        ss = np.exp(r.uniform(math.log(0.1), math.log(10.0), mod.d_out))
        # Exact eigenbasis of E[a a^T] = diag(sa^2): the permutation sorting sa^2 descending.
        pa = np.argsort(-sa ** 2, kind="stable")
        ps = np.argsort(-ss ** 2, kind="stable")
        QA = np.zeros((mod.d_in, mod.d_in)); QA[pa, np.arange(mod.d_in)] = 1.0
        QS = np.zeros((mod.d_out, mod.d_out)); QS[ps, np.arange(mod.d_out)] = 1.0
        if cols_A is not None:
            QA = QA[:, :cols_A]
        if cols_S is not None:
            QS = QS[:, :cols_S]
        return LayerSpec(mod.d_in, mod.d_out, round_to(QA, w.dtype), round_to(QS, w.dtype),
                         np.sort(sa ** 2)[::-1].copy(), np.sort(ss ** 2)[::-1].copy(), sa, ss)
    raise ValueError(w.spectrum)


def layer_inputs(w: Workload, module_index: int, n: int, role_a: int = ROLE_A,
                 role_s: int = ROLE_S, first: int = 0,
                 spec: Optional[LayerSpec] = None) -> Tuple[np.ndarray, np.ndarray]:
    """Activations a [n, T, d_in] and output gradients s [n, T, d_out] of one module for
    examples first..first+n-1, as float32 arrays holding dtype-representable values.

    Each example has its own seed stream, so any subset can be regenerated alone.
    """
    mod = w.modules[module_index]
    a = np.empty((n, w.T, mod.d_in), np.float32)
    s = np.empty((n, w.T, mod.d_out), np.float32)
    for e in range(n):
        ra = rng_for(w.seed, role_a, module_index, first + e)
        rs = rng_for(w.seed, role_s, module_index, first + e)
        av = ra.standard_normal((w.T, mod.d_in)) * w.a_std
        sv = rs.standard_normal((w.T, mod.d_out)) * w.s_std
        if mod.gelu_input:
            av = gelu_exact(av)
        if w.spectrum == "channel":
            if spec is None:
                spec = layer_spec(w, module_index, 1, 1)
            av = av * spec.chan_A[None, :]
            sv = sv * spec.chan_S[None, :]
        a[e] = round_to(av, w.dtype)
        s[e] = round_to(sv, w.dtype)
    return a, s


def random_codes(n: int, words: int, seed: int, role: int = ROLE_CODES) -> np.ndarray:
    """Uniform random sign codes as uint32 words [n, words]."""
    r = rng_for(seed, role)
    return r.integers(0, 2 ** 32, size=(n, words), dtype=np.uint64).astype(np.uint32)


def lognormal_scales(n: int, u: int, sigma: float, seed: int, role: int = ROLE_SCALES) -> np.ndarray:
    r = rng_for(seed, role)
    return np.exp(r.standard_normal((n, u)) * sigma).astype(np.float32)


def first_stage_like(n: int, m: int, seed: int, decay: float = 0.7) -> np.ndarray:
    """Matrix Z [n, m] (float32) with a decaying column spectrum, a stand-in for
    cached first-stage coordinates when fitting the PCA directions."""
    r = rng_for(seed, ROLE_Z)
    col = (np.arange(1, m + 1, dtype=np.float64)) ** (-decay)
    mix = haar_orthogonal(m, rng_for(seed, ROLE_Z, 1)) if m <= 1024 else None
    z = r.standard_normal((n, m)) * col[None, :]
    if mix is not None:
        z = z @ mix.T
    return z.astype(np.float32)


def srht_draw(m: int, k: int, seed: int, module_index: int = 0) -> Tuple[np.ndarray, np.ndarray]:
    """The random parts of one SRHT realisation: m signs (+1 / -1, int8) and k
    distinct rows of the padded width p = 2^ceil(log2 m), drawn uniformly
    without replacement and listed in ascending order (int32)."""
    r = rng_for(seed, ROLE_SRHT, module_index)
    p = 1
    while p < m:
        p *= 2
    signs = np.where(r.integers(0, 2, m) == 1, 1, -1).astype(np.int8)
    rows = np.sort(r.choice(p, size=k, replace=False)).astype(np.int32)
    return signs, rows


def torch_layer_inputs(w: Workload, module_index: int, n: int, device, generator):
    """Device-side inputs (torch RNG) of the same distribution, for runs too large to draw
    on the host. Returns bf16/f32 tensors a [n, T, d_in], s [n, T, d_out]."""
    import torch
    mod = w.modules[module_index]
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    a = torch.randn((n, w.T, mod.d_in), device=device, generator=generator) * w.a_std
    s = torch.randn((n, w.T, mod.d_out), device=device, generator=generator) * w.s_std
    if mod.gelu_input:
        a = torch.nn.functional.gelu(a)
    return a.to(dt), s.to(dt)


def torch_eigvec_rows(d: int, n_rows: int, device, generator, dtype):
    """n_rows orthonormal rows of length d (leading rows of a Haar orthogonal matrix):
    thin QR of a Gaussian d x n_rows matrix on the host, then moved to `device`.
    `generator` is a CPU torch.Generator."""
    import torch
    g = torch.randn((d, n_rows), generator=generator, dtype=torch.float32)
    q, r = torch.linalg.qr(g)
    sgn = torch.sign(torch.diagonal(r))
    sgn[sgn == 0] = 1.0
    q = q * sgn[None, :]
    return q.t().contiguous().to(device=device, dtype=dtype)
