"""The N > 1 path of bench.py on CPU: world_size-2 gloo process groups.

The solve does not shard (replicas only): each rank times its own problem,
the job's time is the slowest rank's (all-reduce MAX after a barrier) and the
whole-job rate counts every rank's units.  The reference arm runs on rank 0
alone; the other ranks exit 0 without work.
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


def _worker(rank, port, times, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE="2", LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=2)
    try:
        ws, r, _ = bench._dist()
        assert (ws, r) == (2, rank)
        dist.barrier()
        ms = bench.max_over_ranks(times[rank], ws, "cpu")
        out[rank] = (ms, bench.whole_job_rate(1000.0, ws, ms))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_whole_job_rate_gloo():
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    times = [3.0, 5.0]                     # rank 1 is the slow one
    mp.start_processes(_worker, args=(port, times, out), nprocs=2, start_method="spawn",
                       join=True)
    for rank in (0, 1):
        ms, rate = out[rank]
        assert ms == 5.0
        assert rate == pytest.approx(2 * 1000.0 / 5e-3)


def test_single_process_is_identity():
    assert bench.max_over_ranks(4.25, 1) == 4.25
    assert bench.whole_job_rate(10.0, 1, 2.0) == pytest.approx(5000.0)


def test_reference_arm_only_on_rank_zero(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")

    class Args:
        config, ref_block, steps, warmup = 2, 8, 1, 0
    assert bench.run_reference(Args()) == 0
    assert capsys.readouterr().out == ""


def test_extra_lines_cpu_baseline_on_small_samples():
    """The oracle leg of the extra bench lines runs on host arrays and reports
    its value in the line's unit (small samples here)."""
    import numpy as np
    import workloads as WL
    rng = np.random.default_rng(0)
    r = bench.extra_cpu_baseline("gram", {"X": rng.normal(size=(64, 32))})
    assert r["unit"] == "flop/s" and r["value"] > 0 and r["kind"] == "oracle"
    r = bench.extra_cpu_baseline("symgrid", {"W": rng.standard_t(4, size=(8, 64))})
    assert r["unit"] == "entries/s" and r["value"] > 0
    W, A, B = WL.small_problem(24, 40, 3)
    f = bench._oracle_factors(A, B, 0.01)
    for wl in ("batched", "gptq"):
        r = bench.extra_cpu_baseline(wl, {"W": W.double().numpy(), "LA": f.LA, "LB": f.LB,
                                          "bits": 4, "rows": W.double().numpy()})
        assert r["unit"] == "entries/s" and r["value"] > 0 and r["cores"] >= 1
    fa = bench._oracle_factors(A, torch.ones(1, 1), 0.01)           # A's factor alone
    np.testing.assert_allclose(fa.LA, f.LA, rtol=1e-12, atol=1e-14)
