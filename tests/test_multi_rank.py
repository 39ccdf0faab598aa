"""The N > 1 path of bench.py on CPU ranks (gloo, world size 2): the step time is the slowest rank's, the
value counts every rank's units, and the reference arm runs on rank 0 alone."""

import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, local_ms, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(local_ms[rank], world, torch.device("cpu"))
        out[rank] = (ms, bench.whole_job_rate(1000, world, ms))
    finally:
        dist.destroy_process_group()


def test_step_time_is_the_slowest_rank_and_value_counts_every_rank():
    world, local_ms = 2, [0.75, 1.25]
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, local_ms, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for r in range(world):
        ms, rate = out[r]
        assert ms == 1.25                                  # both ranks report the maximum
        assert rate == pytest.approx(2 * 1000 / 1.25e-3)   # units of both ranks over the slowest time


def test_reference_arm_runs_on_rank_zero_alone():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2"],
                       env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(0.5, 1, None) == 0.5
    assert bench.whole_job_rate(64, 1, 0.5) == pytest.approx(128000.0)
