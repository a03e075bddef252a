"""Host-side sharding for replicas on several GPUs.

Compression and scoring need no exchange between GPUs: examples are
compressed independently (Alg. 1 stores each example on its own) and each
stored row is scored on its own. A multi-GPU job therefore gives each rank a
contiguous range of examples or stored rows and concatenates the per-rank
results on the host. The only collective is the gather of results.
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
