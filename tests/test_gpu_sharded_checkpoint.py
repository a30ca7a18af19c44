"""Sharded step (gnmr_step_partials on every shard, sums added, gnmr_finish on
every rank) and checkpoint/resume (gnmr_get_state / gnmr_set_state), checked
against the oracle and against an uninterrupted handle."""
import struct

import numpy as np
import pytest

import workloads
from paper_2606_00539_gb300 import Monitor, sharding
from paper_2606_00539_gb300 import _native as N
from tests import trace_driver as TD

pytestmark = pytest.mark.gpu

RTOL = 1e-5


def _monitor(w, off=None, ln=None):
    return Monitor(w.offsets if off is None else off, w.lengths if ln is None else ln, device=0,
                   **w.monitor_kwargs())


@pytest.mark.parametrize("config,shrink,world", [("llama2-13b", 16, 2), ("aq-stress", 8, 3),
                                                 ("moe", 32, 2),
                                                 ("llama2-1.3b", 2, 2)])   # shards with more runs than warps
def test_sharded_step_matches_oracle(config, shrink, world, cuda_device):
    """World-size emulation on one GPU: the ranks' halves run one after the
    other (no kernel waits for another); the all-reduce is a device add."""
    import torch
    w = workloads.make(config, shrink=shrink, steps=12)
    tr = TD.LockstepTrace(w, "cuda:0", _monitor)
    shards = sharding.even_shards(w.arena_elems, world, align=8)
    ranks = []
    for start, n in shards:
        lo, ll = sharding.shard_layout(w.offsets, w.lengths, start, n)
        ranks.append((start, n, _monitor(w, lo, ll)))
    rank_stats = [m.new_stats() for _, _, m in ranks]
    try:
        for t in range(w.steps):
            outs = []

            def sharded_step():
                total = torch.zeros(w.num_units, dtype=torch.float64, device=cuda_device)
                for start, n, m in ranks:
                    total += m.step_partials(tr.arena[start:start + n])
                masks = []
                for (start, n, m), st in zip(ranks, rank_stats):
                    masks.append(m.finish(total, stats=st))
                outs.append(masks)
                # rank 0's outputs are the ones compared with the oracle
                for k in tr.stats:
                    tr.stats[k].copy_(rank_stats[0][k])
                return masks[0]

            norms, res, got = tr.step(t, gpu_step=sharded_step)
            TD.compare(norms, res, got, RTOL)
            m0 = outs[0][0].cpu()
            for r in range(1, world):
                assert np.array_equal(outs[0][r].cpu().numpy(), m0.numpy())
                for k in rank_stats[0]:
                    assert torch.equal(rank_stats[r][k], rank_stats[0][k]), k
    finally:
        tr.close()
        for _, _, m in ranks:
            m.close()


def _parse_blob(blob, U, window):
    magic, version, nu, win, steps, _ = struct.unpack_from("<4sIiiqq", blob, 0)
    assert magic == b"GNMR" and version == 2 and nu == U and win == window
    rec = np.frombuffer(blob, dtype=np.dtype([("A", "<f8"), ("k", "<i8"), ("fill", "<i4"),
                                              ("head", "<i4"), ("lock", "<i4"), ("active", "<i4"),
                                              ("gsum", "<f8")]),
                        count=U, offset=32)
    q = np.frombuffer(blob, dtype="<f8", count=U * window, offset=32 + 40 * U).reshape(U, window)
    return steps, rec, q


def test_checkpoint_blob_matches_oracle_state(cuda_device):
    w = workloads.make("tiny", seed=4, steps=30, shrink=2)
    tr = TD.LockstepTrace(w, "cuda:0", _monitor)
    try:
        for t in range(17):
            norms, res, got = tr.step(t)
            TD.compare(norms, res, got, RTOL)
        blob = tr.mon.get_state()
        steps, rec, q = _parse_blob(blob, w.num_units, w.window)
        st = tr.ctl.get_state()
        assert steps == st["t"] == 17
        np.testing.assert_allclose(rec["A"], st["A"], rtol=RTOL)
        assert np.array_equal(rec["k"], st["k"])
        assert np.array_equal(rec["fill"], st["qlen"])
        assert np.array_equal(rec["lock"], st["lock"])
        assert np.array_equal(rec["active"], tr.ctl.policy_state()["active"])
        for b in range(w.num_units):        # ring (oldest at head) vs oldest-first list
            n = rec["fill"][b]
            ring = np.roll(q[b], -rec["head"][b])[:n] if n == w.window else q[b][:n]
            np.testing.assert_allclose(ring, st["Q"][b][:n], rtol=RTOL)
    finally:
        tr.close()


def test_resume_continues_the_trace_exactly(cuda_device):
    import torch
    w = workloads.make("llama2-13b", shrink=32, steps=14)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    a = _monitor(w)
    sa = a.new_stats()
    try:
        for t in range(6):
            f.fill(arena, t)
            a.step(arena, stats=sa)
        blob = a.get_state()
        b = _monitor(w)
        sb = b.new_stats()
        b.set_state(blob)
        assert b.info()["steps"] == 6
        for t in range(6, w.steps):
            f.fill(arena, t)
            ma = a.step(arena, stats=sa)
            mb = b.step(arena, stats=sb)
            assert torch.equal(ma, mb)
            for k in sa:
                assert torch.equal(sa[k], sb[k]), k
        assert b.get_state() == a.get_state()
        b.close()
    finally:
        a.close()


def test_set_state_rejects_bad_blobs(cuda_device):
    w = workloads.make("tiny", steps=3, shrink=8)
    a = _monitor(w)
    other = Monitor(w.offsets[:10], w.lengths[:10], device=0, **dict(w.monitor_kwargs(),
                                                                     recoverable=None))
    try:
        good = a.get_state()
        bad_magic = b"XXXX" + good[4:]
        truncated = good[:-8]
        bad_lock = bytearray(good)
        struct.pack_into("<i", bad_lock, 32 + 24, 99)          # unit 0's lock > T_lock
        for blob in (bad_magic, truncated, bytes(bad_lock), other.get_state()):
            with pytest.raises(N.GnmrError) as ei:
                a.set_state(blob)
            assert ei.value.status == N.GNMR_ERR_INVALID_ARG
        a.set_state(good)                                       # still usable
    finally:
        a.close()
        other.close()


def test_sharded_step_helper_over_a_one_rank_nccl_group(cuda_device):
    """sharding.sharded_step with a real process group (NCCL, one rank: the
    shard is the whole arena and the all-reduce an identity) gives the
    masks, locks and norms of a plain gnmr_step handle."""
    import os
    import socket
    import torch
    import torch.distributed as dist
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("nccl", rank=0, world_size=1, device_id=cuda_device)
    w = workloads.make("tiny", steps=10)
    f = workloads.Filler(w, cuda_device)
    arena = f.new_arena()
    plain, sharded = _monitor(w), _monitor(w)
    sp, ss = plain.new_stats(), sharded.new_stats()
    try:
        for t in range(w.steps):
            f.fill(arena, t)
            m1 = plain.step(arena, stats=sp)
            m2 = sharding.sharded_step(sharded, arena, stats=ss)
            torch.cuda.synchronize()
            assert torch.equal(m1, m2), f"step {t + 1}: mask"
            assert torch.equal(sp["lock"], ss["lock"]), f"step {t + 1}: lock"
            np.testing.assert_allclose(ss["norm"].cpu().numpy(), sp["norm"].cpu().numpy(), rtol=1e-12, atol=0)
    finally:
        plain.close()
        sharded.close()
        dist.destroy_process_group()
