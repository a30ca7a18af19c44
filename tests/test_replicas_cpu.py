"""Multi-process path of bench.py on CPU (gloo, world size 2): the max over
ranks, the barrier and the whole-job throughput; the reference arm does its
work on rank 0 only.  On one replica the monitor has no exchange step, so
replicas are independent and only timing is aggregated."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    local_ms = [120.0, 150.0][rank]
    bench.barrier(world)
    mx = bench.max_over_ranks(local_ms, world)
    value = bench.throughput_gbs(world, 25_375_539_200, 10, mx)
    out.put((rank, mx, value))
    dist.destroy_process_group()


def test_max_over_ranks_and_throughput_gloo():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    mp.start_processes(_worker, args=(world, port, q), nprocs=world, join=True,
                       start_method="spawn")
    got = sorted(q.get(timeout=60) for _ in range(world))
    for rank, mx, value in got:
        assert mx == 150.0
        assert value == pytest.approx(2 * 25_375_539_200 * 10 / 0.150 / 1e9)


def test_reference_arm_other_ranks_do_nothing(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    bench.run_reference(bench.parse_args(["--impl", "reference", "--steps", "1", "--warmup", "0"]))
    assert capsys.readouterr().out == ""


def test_single_rank_helpers_are_identities():
    assert bench.max_over_ranks(3.5, 1) == 3.5
    bench.barrier(1)
    assert bench.throughput_gbs(1, 10**9, 1, 1000.0) == pytest.approx(1.0)
