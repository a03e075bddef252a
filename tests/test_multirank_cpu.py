"""Replica sharding across ranks, as a gloo world of 2 on CPU.

Each rank scores its contiguous shard of a synthetic store with the oracle;
the gathered scores must equal the unsharded scores exactly, and the job-level
timing reduction (max over ranks) must match bench.py's rule. The sharded PCA
fit (one all-reduce of the second moment) is run with the oracle's arithmetic
in place of the device calls and must equal the fit on all rows."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out_dir):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import torch.distributed as dist

    from oracle import eogp_oracle as O
    from paper_2609_37842_gb300.shard import all_gather_rows, shard_range
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    rng = np.random.default_rng(5)
    ks = [64, 40, 128]
    N, Q = 37, 5
    tc = O.pack_concat([rng.integers(0, 2, (N, k)).astype(bool) for k in ks])
    qc = O.pack_concat([rng.integers(0, 2, (Q, k)).astype(bool) for k in ks])
    ts = rng.lognormal(0, 0.5, (N, 3)).astype(np.float32)
    qs = rng.lognormal(0, 0.5, (Q, 3)).astype(np.float32)
    lo, hi = shard_range(N, rank, world)
    local = O.score_codes_f32(tc[lo:hi], ts[lo:hi], ks, qc, qs).T   # rows = stored examples
    allrows = all_gather_rows(torch.from_numpy(np.ascontiguousarray(local)), N, world)
    # sharded PCA fit: each rank's rows, one reduction of the second moment
    from paper_2609_37842_gb300.shard import fit_pca_sharded
    Z = np.random.default_rng(9).standard_normal((41, 10)) * np.linspace(2, 0.3, 10)[None, :]
    zlo, zhi = shard_range(41, rank, world)
    Pt_sh, mu_sh = fit_pca_sharded(torch.from_numpy(Z[zlo:zhi]), 4,
                                   moment_fn=lambda z: torch.from_numpy(z.numpy().T @ z.numpy()),
                                   fit_fn=lambda C, n, k: O.fit_pca_from_moment(C.numpy(), n, k))
    # per-rank step time -> job time = max over ranks (bench.py's rule)
    t = torch.tensor([10.0 + rank])
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    if rank == 0:
        np.save(os.path.join(out_dir, "sharded.npy"), allrows.numpy().T)
        np.save(os.path.join(out_dir, "full.npy"), O.score_codes_f32(tc, ts, ks, qc, qs))
        np.save(os.path.join(out_dir, "tmax.npy"), t.numpy())
        np.save(os.path.join(out_dir, "pca_sharded.npy"), Pt_sh)
        np.save(os.path.join(out_dir, "pca_full.npy"), O.fit_pca(Z, 4, route="cov")[0])
    dist.barrier()
    dist.destroy_process_group()


def test_sharded_scores_equal_unsharded(tmp_path):
    import torch.multiprocessing as mp
    world = 2
    mp.spawn(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    sharded = np.load(tmp_path / "sharded.npy")
    full = np.load(tmp_path / "full.npy")
    np.testing.assert_array_equal(sharded, full)
    assert float(np.load(tmp_path / "tmax.npy")[0]) == 11.0
    np.testing.assert_allclose(np.load(tmp_path / "pca_sharded.npy"), np.load(tmp_path / "pca_full.npy"),
                               atol=1e-10)


def test_shard_range_covers_exactly():
    from paper_2609_37842_gb300.shard import shard_range
    for n in (0, 1, 7, 37, 1000):
        for world in (1, 2, 3, 8):
            spans = [shard_range(n, r, world) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
            sizes = [h - l for l, h in spans]
            assert max(sizes) - min(sizes) <= 1
