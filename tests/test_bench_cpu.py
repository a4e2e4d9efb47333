"""CPU checks of bench.py's multi-rank logic (replicas: one independent PS per
GPU, the slowest rank sets the job time) with two gloo ranks, and of the
reference arm's rank handling."""
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        times = [10.0 * (rank + 1), 0.5 + rank]            # rank 1 is the slow one
        got = bench.combine_over_ranks(times, world, "cpu")
        out[rank] = got + [bench.job_value(world, 20, got[0])]
    finally:
        dist.destroy_process_group()


def test_combine_over_ranks_takes_the_slowest_rank():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, port, out), nprocs=world, join=True, start_method="spawn")
    for r in range(world):
        elapsed, e2e, value = out[r]
        assert elapsed == 20.0 and e2e == 1.5
        assert value == pytest.approx(2 * 20 / 0.020)


def test_single_rank_combine_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.combine_over_ranks([3.0, 4.0], 1, "cpu") == [3.0, 4.0]
    assert bench.job_value(1, 10, 100.0) == pytest.approx(100.0)


def test_reference_arm_nonzero_rank_exits_quietly():
    env = dict(os.environ, WORLD_SIZE="2", RANK="1", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "3",
                        "--warmup", "3"], capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""
