"""The N>1 host path of bench.py on CPU: two gloo ranks, replicas timed by the
slowest rank, whole-job rate summed over ranks (no GPU involved)."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = [4.0, 7.5][rank]
        ms = bench.max_over_ranks(local_ms)
        rate = bench.whole_job_rate(world, 1000, ms)
        q.put((rank, ms, rate))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for rank, ms, rate in got:
        assert ms == pytest.approx(7.5)
        assert rate == pytest.approx(2 * 1000 / 7.5e-3)


def test_single_process_needs_no_group():
    assert bench.max_over_ranks(3.0) == 3.0
    assert bench.whole_job_rate(1, 10, 2.0) == pytest.approx(5000.0)
