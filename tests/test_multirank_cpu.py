"""The benchmark's multi-rank logic (one replica of the workload per rank,
weak scaling) on two CPU ranks over gloo: the barrier, the max-over-ranks
timing and the whole-job throughput formula."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench.barrier(world)
        times = [0.010, 0.025]          # the second rank is the slower one
        t = bench.max_over_ranks(times[rank], world, device="cpu")
        rate = bench.whole_job_rate(1.0e9, world, t)
        shard_bytes = [4.0e8, 4.2e8]    # the shards keep slightly different rows
        total = bench.sum_over_ranks(shard_bytes[rank], world, device="cpu")
        out[rank] = (t, rate, total)
        bench.barrier(world)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_sum_the_work():
    world = 2
    port = _free_port()
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    for r in range(world):
        t, rate, total = out[r]
        assert t == pytest.approx(0.025)
        assert rate == pytest.approx(2 * 1.0e9 / 0.025)
        assert total == pytest.approx(8.2e8)


def test_single_rank_is_the_identity():
    import bench
    assert bench.max_over_ranks(0.5, 1) == 0.5
    assert bench.sum_over_ranks(0.5, 1) == 0.5
    assert bench.whole_job_rate(3.0, 1, 1.5) == pytest.approx(2.0)
