"""GB300 (sm_103a) implementation of the EOGP hot path: one-bit gradient
compression (Kronecker-eigenbasis first stage, PCA second stage, sign packing)
and influence scoring against stored codes, behind the C ABI in include/eogp.h.

`eogp` is the ctypes binding; `build` compiles libeogp.so in-tree; `synth`
draws seeded synthetic workloads.
"""
from . import build  # noqa: F401
from . import eogp  # noqa: F401

__all__ = ["eogp", "build"]
