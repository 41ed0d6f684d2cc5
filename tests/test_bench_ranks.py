"""Host-side check of the benchmark's multi-rank aggregation (no GPU): two gloo ranks on the CPU
each report their own timed-region duration; both must see the slowest one, and the whole-job
rate must count the units of every rank over that time."""
import os
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 100.0 + 25.0 * rank            # rank 1 is the slower one
        t_max = bench.max_over_ranks(local_ms, torch.device("cpu"), world)
        rate = bench.whole_job_rate(512, 10, world, t_max)
        out[rank] = (t_max, rate)
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_rate_gloo_world2():
    world = 2
    port = 29500 + (os.getpid() % 1000)
    with mp.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
        res = dict(out)
    assert set(res) == {0, 1}
    for r in range(world):
        t_max, rate = res[r]
        assert t_max == 125.0
        assert rate == pytest.approx(512 * 10 * world / 0.125)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, torch.device("cpu"), 1) == 3.5
    assert bench.whole_job_rate(100, 4, 1, 2.0) == pytest.approx(200000.0)
