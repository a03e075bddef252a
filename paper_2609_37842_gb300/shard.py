"""Host-side sharding for replicas on several GPUs.

Compression and scoring need no exchange between GPUs: examples are
compressed independently (Alg. 1 stores each example on its own) and each
stored row is scored on its own. A multi-GPU job therefore gives each rank a
contiguous range of examples or stored rows and concatenates the per-rank
results on the host. The PCA fit over rows held by several ranks needs one
reduction: the m x m second moment summed over the ranks (App. B.2, the
covariance route), after which every rank fits the same P.
"""
from __future__ import annotations

from typing import Tuple


def shard_range(n: int, rank: int, world: int) -> Tuple[int, int]:
    """Contiguous [lo, hi) range of n items for `rank` of `world`; sizes differ by at most 1."""
    if world < 1 or not (0 <= rank < world) or n < 0:
        raise ValueError("bad shard arguments")
    base, extra = divmod(n, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def all_gather_rows(local, n_total: int, world: int, group=None):
    """Concatenate every rank's rows (dim 0, ranges from shard_range) on every rank.

    Uneven shards are padded to the largest shard for the collective and trimmed
    afterwards. Works with any torch.distributed backend (gloo on CPU tensors)."""
    import torch
    import torch.distributed as dist
    sizes = [shard_range(n_total, r, world)[1] - shard_range(n_total, r, world)[0]
             for r in range(world)]
    width = max(sizes)
    pad = torch.zeros((width,) + tuple(local.shape[1:]), dtype=local.dtype, device=local.device)
    pad[:local.shape[0]] = local
    bufs = [torch.empty_like(pad) for _ in range(world)]
    dist.all_gather(bufs, pad, group=group)
    return torch.cat([b[:s] for b, s in zip(bufs, sizes)], dim=0)


def fit_pca_sharded(Z_local, k: int, group=None, moment_fn=None, fit_fn=None):
    """PCA directions from rows spread over the ranks of `group` (App. B.2,
    covariance route): every rank adds its rows' second moment Z_s^T Z_s, one
    all-reduce sums the m x m fp64 matrices (and the row counts), and every rank
    fits P from the sum. moment_fn(Z) -> C and fit_fn(C, n_total, k) -> (Pt, eig)
    default to the library calls eogp_second_moment / eogp_fit_pca_from_moment;
    the reduction goes through host memory for CPU backends (gloo)."""
    import torch
    import torch.distributed as dist
    if moment_fn is None or fit_fn is None:
        from . import eogp as E
        moment_fn = moment_fn or (lambda Z: E.second_moment(Z))
        fit_fn = fit_fn or (lambda C, n, kk: E.fit_pca_from_moment(C, n, kk))
    C = moment_fn(Z_local)
    n = torch.tensor([float(Z_local.shape[0])], dtype=torch.float64)
    if dist.is_available() and dist.is_initialized():
        on_host = dist.get_backend(group) == "gloo"
        red = C.cpu() if on_host else C
        dist.all_reduce(red, group=group)
        C = red.to(C.device) if on_host else red
        if not on_host:
            n = n.to(C.device)
        dist.all_reduce(n, group=group)
    return fit_fn(C, int(n.item()), k)
