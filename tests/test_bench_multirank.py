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


def test_host_link_bytes_counts_the_defined_slots():
    """Two layers, two sequences: the rows entering each layer go in (Q, K, V),
    their O rows and scores come back, pos for every layer and len."""
    import bench
    lens = [[5, 3], [2, 3], [1, 0]]       # len[l][b], l = 0..2
    H, d = 2, 64
    row = H * d * 2                       # one bf16 row of one tensor
    h2d, d2h = bench.host_link_bytes(lens, 2, H, d, mask_bytes=16)
    entering = 5 + 3 + 2 + 3              # layers 0 and 1
    assert h2d == 3 * row * entering + 16
    assert d2h == entering * (row + 4) + 4 * (5 + 3 + 2 + 3 + 1 + 0) + 4 * 6
