"""Multi-process host logic of bench.py's N-replica mode, on CPU with gloo.

The path does not shard (one independent replica per GPU), so the only
cross-rank steps are the timing reduction (the slowest rank's time) and the
whole-job throughput; both are checked here with two ranks.
"""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, _ = bench.dist_env()
        assert (w, r) == (world, rank)
        # rank r took (r + 1) * 10 ms per step: the job is as slow as its slowest rank
        ms = bench.max_over_ranks((rank + 1) * 10.0, world, torch)
        out[rank] = (ms, bench.job_throughput(8192, world, ms / 1e3))
    finally:
        dist.destroy_process_group()


def test_two_replicas_report_slowest_rank_and_job_throughput():
    world = 2
    out = mp.Manager().dict()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, start_method="spawn")
    for rank in range(world):
        ms, tput = out[rank]
        assert ms == 20.0
        assert tput == pytest.approx(8192 * 2 / 0.020)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(12.5, 1, torch) == 12.5
    assert bench.job_throughput(1000, 1, 0.5) == 2000.0
