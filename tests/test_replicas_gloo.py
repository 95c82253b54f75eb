"""The multi-GPU path is replicas only (independent image batches, replicated
weights): ranks meet at the timing barrier and a max-reduce of the step time.
This checks that host logic with two gloo ranks on the CPU."""
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


def _rank(rank, world, port, local_ms, images, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        ms = bench.job_step_time(local_ms[rank], dist, torch.device("cpu"))
        value = bench.job_throughput(images, world, ms)
        dist.barrier()
        out.put((rank, ms, value, bench.replica_seed(1000, rank)))
    finally:
        dist.destroy_process_group()


def test_two_replicas_report_the_slowest_rank_and_the_whole_job():
    world, images = 2, 8
    local_ms = [10.0, 12.5]
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, local_ms, images, out)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, value, seed in res:
        assert ms == pytest.approx(12.5)                       # max over ranks
        assert value == pytest.approx(world * images / 0.0125)  # all images over the slowest step
    assert res[0][3] != res[1][3]                               # each replica draws its own inputs


def test_single_process_needs_no_collective():
    assert bench.job_step_time(7.0) == 7.0
    assert bench.job_throughput(8, 1, 40.0) == pytest.approx(200.0)
