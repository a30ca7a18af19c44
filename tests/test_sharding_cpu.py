"""Host logic of the sharded step on CPU: shard layouts cover every unit's
elements exactly once, and per-rank sums of squares all-reduced over gloo
(world size 2) give the full-arena norms of Eq. local_gradient."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

import oracle
from paper_2606_00539_gb300 import sharding as S


def _layout(rng, U=300):
    ln = rng.integers(0, 5000, U).astype(np.int64)
    off = np.concatenate([[0], np.cumsum(ln)[:-1]]).astype(np.int64) + rng.integers(0, 3, U)
    return off, ln


@pytest.mark.parametrize("world,align", [(1, 1), (2, 1), (3, 8), (7, 256)])
def test_shards_partition_every_unit(world, align):
    rng = np.random.default_rng(world)
    off, ln = _layout(rng)
    total = int((off + ln).max())
    shards = S.even_shards(total, world, align)
    assert sum(n for _, n in shards) == total
    assert shards[0][0] == 0 and all(shards[i][0] + shards[i][1] == shards[i + 1][0]
                                     for i in range(world - 1))
    covered = np.zeros(len(off), np.int64)
    for start, n in shards:
        lo, ll = S.shard_layout(off, ln, start, n)
        assert np.all(lo >= 0) and np.all(lo + ll <= max(n, 0))
        covered += ll
    assert np.array_equal(covered, ln)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, arena, off, ln, q):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    start, n = S.even_shards(len(arena), world)[rank]
    lo, ll = S.shard_layout(off, ln, start, n)
    local = arena[start:start + n].astype(np.float64)
    sums = np.array([np.sum(local[o:o + k] ** 2) for o, k in zip(lo, ll)])
    t = torch.from_numpy(sums)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    q.put((rank, np.sqrt(t.numpy())))
    dist.destroy_process_group()


def test_sharded_norms_over_gloo():
    rng = np.random.default_rng(5)
    off, ln = _layout(rng, 120)
    arena = rng.standard_normal(int((off + ln).max()) + 10).astype(np.float32)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    mp.start_processes(_rank, args=(2, _free_port(), arena, off, ln, q), nprocs=2, join=True,
                       start_method="spawn")
    got = dict(q.get(timeout=60) for _ in range(2))
    want = oracle.unit_norms(arena, off, ln)
    for r in (0, 1):
        np.testing.assert_allclose(got[r], want, rtol=1e-12, atol=0)
    assert np.array_equal(got[0], got[1])        # every rank sees the same sums
