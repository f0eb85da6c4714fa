"""The benchmark's multi-rank aggregation on CPU: two gloo ranks, each a
replica with its own timings; every rank ends with the slowest rank's
timings, and the whole-job throughput counts both replicas' work over that
time."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = [1.0 + rank, 5.0 - rank, 0.25 * (rank + 1)]  # gemm ms, e2e ms, wall s
        out[rank] = bench.max_over_ranks(mine, world, torch.device("cpu"))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_ranks_take_the_slowest_timings():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(100)
            assert p.exitcode == 0
        assert out[0] == out[1] == [2.0, 5.0, 0.5]


def test_single_rank_and_whole_job_value():
    assert bench.max_over_ranks([3.0, 0.0, 1.5], 1, torch.device("cpu")) == [3.0, 0.0, 1.5]
    # two replicas of 2 * 4096^3 operations each, slowest rank 0.1 ms
    ops = 2 * 4096 ** 3
    assert bench.whole_job_tops(ops, 2, 0.1) == pytest.approx(2 * ops / 1e-4 / 1e12)
    assert bench.whole_job_tops(ops, 1, 0.1) == pytest.approx(ops / 1e-4 / 1e12)
