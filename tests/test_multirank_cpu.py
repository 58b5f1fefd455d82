"""The multi-GPU path on CPU: two gloo ranks, as bench.py runs them under
torchrun (one process per GPU, each on its own token batch, no collective
on the data path).  The only cross-rank step is the timing reduction: the
job time is the slowest rank's, and the job rate counts every rank's work.
Also: each rank's batch has the workload's shape but its own values, and the
reference arm prints nothing on ranks other than 0."""
import contextlib
import io
import json
import os
import socket
import sys

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = [40.0, 50.0][rank]  # rank 1 is the slower one
        ms, tops = bench.job_throughput(local_ms, 1e12, 10, world)
        out[rank] = (ms, tops)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_count_all_work():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_rank_main, args=(world, port, out), nprocs=world,
                           join=True, start_method="spawn")
        res = dict(out)
    assert set(res) == {0, 1}
    for rank in (0, 1):
        ms, tops = res[rank]
        assert ms == 50.0
        # 2 ranks x 10 steps x 1e12 operations in 50 ms
        assert abs(tops - 2 * 10 * 1e12 / 0.05 / 1e12) < 1e-9


def test_single_rank_needs_no_process_group():
    import bench
    ms, tops = bench.job_throughput(25.0, 2e12, 4, 1)
    assert ms == 25.0 and abs(tops - 2e12 * 4 / 0.025 / 1e12) < 1e-9


def test_each_rank_gets_its_own_batch():
    from paper_2509_24416_gb300 import synth
    cfg = dict(synth.WORKLOADS["single_1152"], M=32)
    d0 = synth.layer_inputs(cfg, 0, batch=0)
    d1 = synth.layer_inputs(cfg, 0, batch=1)
    assert d0["X"].shape == d1["X"].shape == (32, 1152)
    assert not np.array_equal(d0["X32"], d1["X32"])
    assert np.array_equal(d0["W32"], d1["W32"])        # replicated weights
    assert np.array_equal(d0["calib"], d1["calib"])    # same swap vector


def test_reference_arm_is_silent_on_other_ranks(monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    args = bench.parse()
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.reference_arm(args)
    assert buf.getvalue() == ""
