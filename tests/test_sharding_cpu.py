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


def _controller_rank(rank, world, port, arenas, off, ln, q):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    start, n = S.even_shards(len(arenas[0]), world)[rank]
    lo, ll = S.shard_layout(off, ln, start, n)
    ctl = oracle.Controller(len(off), window=3, max_o=2, lock_len=2, alpha=(1.5, 1.2), beta=(1.4, 1.4),
                            warmup_steps=2)
    out = []
    try:
        for arena in arenas:
            local = arena[start:start + n].astype(np.float64)
            t = torch.from_numpy(np.array([np.sum(local[o:o + k] ** 2) for o, k in zip(lo, ll)]))
            dist.all_reduce(t, op=dist.ReduceOp.SUM)
            res = ctl.step(np.sqrt(t.numpy()))
            out.append((res.mask.copy(), res.lock.copy()))
    finally:
        ctl.close()
    q.put((rank, out))
    dist.destroy_process_group()


def test_sharded_controller_gives_every_rank_the_same_decisions():
    """The sharded step: each rank reduces its slice of every unit, the sums
    are all-reduced, and every rank steps the same deterministic controller
    (Algorithms 1-2) -- so the masks and locks agree across ranks and with an
    unsharded controller on the whole arena."""
    rng = np.random.default_rng(11)
    off, ln = _layout(rng, 40)
    total = int((off + ln).max()) + 7
    scale = np.exp(rng.normal(0.0, 1.0, len(off)))
    arenas = []
    for t in range(8):
        s = scale.copy()
        s[rng.choice(len(off), 3, replace=False)] *= rng.uniform(5.0, 50.0, 3)   # spikes
        a = np.zeros(total, np.float32)
        for b, (o, k) in enumerate(zip(off, ln)):
            a[o:o + k] = rng.standard_normal(k) * s[b]
        arenas.append(a)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    mp.start_processes(_controller_rank, args=(2, _free_port(), arenas, off, ln, q), nprocs=2,
                       join=True, start_method="spawn")
    got = dict(q.get(timeout=60) for _ in range(2))
    ref = oracle.Controller(len(off), window=3, max_o=2, lock_len=2, alpha=(1.5, 1.2), beta=(1.4, 1.4),
                            warmup_steps=2)
    try:
        selected = 0
        for t, arena in enumerate(arenas):
            res = ref.step(oracle.unit_norms(arena, off, ln))
            selected += int(res.mask.sum())
            for r in (0, 1):
                assert np.array_equal(got[r][t][0], got[0][t][0]) and np.array_equal(got[r][t][1], got[0][t][1])
                assert np.array_equal(got[r][t][0], res.mask), f"step {t + 1}, rank {r}: mask"
                assert np.array_equal(got[r][t][1], res.lock), f"step {t + 1}, rank {r}: lock"
        assert selected > 0                          # the spikes were selected at some step
    finally:
        ref.close()


class _RecordingMonitor:
    """Stands in for Monitor on CPU: its partial sums are the rank's local
    sums of squares, and finish records what it was given."""

    def __init__(self, arena, lo, ll):
        self.arena, self.lo, self.ll = arena, lo, ll
        self.finished = None

    def step_partials(self, local_arena, sumsq=None):
        import torch
        local = local_arena.numpy().astype(np.float64)
        return torch.tensor([np.sum(local[o:o + k] ** 2) for o, k in zip(self.lo, self.ll)],
                            dtype=torch.float64)

    def finish(self, sums, mask=None, stats=None):
        self.finished = sums.numpy().copy()
        return "mask"


def _helper_rank(rank, world, port, arena, off, ln, q):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    start, n = S.even_shards(len(arena), world)[rank]
    lo, ll = S.shard_layout(off, ln, start, n)
    mon = _RecordingMonitor(arena, lo, ll)
    out = S.sharded_step(mon, torch.from_numpy(arena[start:start + n].copy()))
    q.put((rank, out, mon.finished))
    dist.destroy_process_group()


def test_sharded_step_helper_finishes_on_the_summed_sums():
    rng = np.random.default_rng(21)
    off, ln = _layout(rng, 50)
    arena = rng.standard_normal(int((off + ln).max()) + 3).astype(np.float32)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    mp.start_processes(_helper_rank, args=(2, _free_port(), arena, off, ln, q), nprocs=2, join=True,
                       start_method="spawn")
    got = dict((r, (out, fin)) for r, out, fin in (q.get(timeout=60) for _ in range(2)))
    want = oracle.unit_norms(arena, off, ln) ** 2
    for r in (0, 1):
        assert got[r][0] == "mask"
        np.testing.assert_allclose(got[r][1], want, rtol=1e-12, atol=1e-300)
    assert np.array_equal(got[0][1], got[1][1])
