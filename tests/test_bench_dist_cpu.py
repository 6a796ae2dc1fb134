"""The multi-process path of bench.py on CPU: two gloo ranks (127.0.0.1) reduce their
step times to the slowest one, and the whole-job rate counts every rank's work over that
time; the reference arm does its work on rank 0 only."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        local_ms = [3.0, 5.0][rank]
        out[rank] = bench.max_over_ranks(local_ms, world, "cpu")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time():
    world, port = 2, _free_port()
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    assert out[0] == out[1] == 5.0


def test_whole_job_rate_counts_all_ranks():
    # 2 ranks x 10 TFLOP each over the slowest rank's 0.5 s = 40 TFLOP/s
    assert bench.whole_job_tflops(2, 10e12, 0.5) == pytest.approx(40.0)
    assert bench.whole_job_tflops(1, 10e12, 0.5) == pytest.approx(20.0)
    assert bench.max_over_ranks(7.5, 1) == 7.5


def test_reference_arm_runs_on_rank_zero_only(capsys):
    ns = type("A", (), dict(gpus=2, steps=1, warmup=1, impl="reference", layers=1, e2e_steps=0,
                            no_cpu_baseline=True))()
    bench.run_reference(ns, rank=1)
    assert capsys.readouterr().out == ""


def test_launch_count_of_the_mask_build():
    assert bench.mask_launches(64, 64) == 1
    assert bench.mask_launches(64, 256) == 1
    assert bench.mask_launches(64, 289) == 2
    assert bench.mask_launches(128, 64) == 2
