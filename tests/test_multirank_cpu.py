"""The multi-process path of the benchmark on CPU: world size 2 over gloo.

Under torchrun every rank routes its own replica of the workload (the routing decision of
one batch runs on one GPU); the job's time is the slowest rank's and its rate counts every
rank's requests.  These tests run the reduction bench.py uses, on CPU ranks.
"""

import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, times, out):
    import torch.distributed as dist

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(times[rank], dist, "cpu")
        out[rank] = (ms, bench.whole_job_rate(1000, world, 4, ms))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("times", [(2.0, 5.0), (7.5, 1.25)])
def test_two_ranks_take_the_slowest_time_and_count_every_rank(times):
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        procs = [ctx.Process(target=_rank, args=(r, world, port, times, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    slowest = max(times)
    for r in range(world):
        ms, rate = res[r]
        assert ms == slowest
        # 2 ranks x 1000 requests x 4 steps over the slowest rank's time
        assert rate == pytest.approx(2 * 1000 * 4 / (slowest / 1e3))


def test_single_process_is_the_identity():
    assert bench.max_over_ranks(3.25, None, "cpu") == 3.25
    assert bench.whole_job_rate(65536, 1, 20, 20.0) == pytest.approx(65536 * 20 / 0.02)
