"""Host-side logic of the N>1 benchmark, run as world-size-2 `gloo` ranks on the CPU.

The path shards into independent replicas (one per GPU, no data-path collective); the only
cross-rank steps are the timing reductions: every rank's step, end-to-end and warm-cache
times are reduced with a maximum (the job is as slow as its slowest replica) and the
whole-job throughput is the work all ranks did over that time.  Under torchrun the
reference arm runs on rank 0 alone; the other ranks exit 0 without work or output.
"""
from __future__ import annotations

import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, times, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        got = bench.max_over_ranks(times[rank], world)
        out[rank] = got
        torch.distributed.barrier()
    finally:
        torch.distributed.destroy_process_group()


def test_max_over_ranks_two_gloo_ranks():
    times = [3.25, 7.5]
    port = _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    mp.start_processes(_rank_main, args=(2, port, times, out), nprocs=2, join=True, start_method="spawn")
    assert out[0] == out[1] == max(times)


def test_max_over_ranks_single_rank_is_identity():
    assert bench.max_over_ranks(4.5, 1) == 4.5


def test_job_throughput_counts_every_rank():
    # 2 ranks x 10 steps x 3 units per rank-step over the slowest rank's 5 s
    assert bench.job_throughput(3.0, 2, 10, 5.0) == pytest.approx(12.0)
    # weak scaling: per-rank work fixed, the aggregate grows with the world size
    one = bench.job_throughput(3.0, 1, 10, 5.0)
    assert bench.job_throughput(3.0, 4, 10, 5.0) == pytest.approx(4 * one)


def test_reference_arm_non_zero_rank_exits_quietly():
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2",
               MASTER_ADDR="127.0.0.1", MASTER_PORT=str(_free_port()))
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "1", "--warmup", "3"],
                       env=env, capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""
