"""bench.py's multi-rank host logic on CPU: two gloo ranks, the same helpers
bench uses under torchrun/NCCL.  The slowest rank sets the job time, and the
job value counts every rank's work (weak scaling of independent replicas)."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, local_ms, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        job_ms = bench.max_over_ranks(local_ms[rank], world, torch.device("cpu"))
        out.put((rank, job_ms, bench.job_tflops(2e12, 10, job_ms, world)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_job_time_is_max_over_ranks_and_value_counts_all_ranks(world):
    local_ms = [4.0 + rank for rank in range(world)]   # the last rank is the slowest
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    mp.start_processes(_worker, args=(world, _free_port(), local_ms, out), nprocs=world,
                       join=True, start_method="spawn")
    got = sorted(out.get(timeout=60) for _ in range(world))
    slowest = max(local_ms)
    for rank, job_ms, tflops in got:
        assert job_ms == slowest
        assert tflops == pytest.approx(world * 2e12 * 10 / (slowest * 1e-3) / 1e12)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert not dist.is_initialized()
    assert bench.max_over_ranks(7.5, 1, torch.device("cpu")) == 7.5
    assert bench.job_tflops(1e12, 4, 2.0, 1) == pytest.approx(2000.0)


def test_reference_arm_runs_on_rank_zero_only():
    """Under torchrun the reference arm runs on rank 0; other ranks exit
    without work (no oracle call, no output line)."""
    import argparse
    sys.path.insert(0, ROOT)
    import bench
    assert bench.run_reference(argparse.Namespace(config=2, steps=1, warmup=0), 1) is None
