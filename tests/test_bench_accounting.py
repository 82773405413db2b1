"""CPU checks of bench.py's accounting: the algorithmic flop count F_alg, the
peak it is divided by, and the claim that the oracle's top-left-block sample
is an exact piece of the full solve."""
import numpy as np
import pytest

import bench
import oracle as O
import workloads as WL


def test_f_alg_matches_the_tabulated_values():
    # 2 x the multiply-adds with structurally nonzero factor operands of Alg. 4
    # down to single entries (cheaper order, strictly-lower triangular parts)
    assert bench.f_alg(128, 128) == pytest.approx(7.168e6, rel=1e-3)
    assert bench.f_alg(4096, 4096) == pytest.approx(2.403e11, rel=1e-3)
    assert bench.f_alg(11008, 4096) == pytest.approx(1.081e12, rel=1e-3)
    assert bench.f_alg(4096, 11008) == pytest.approx(1.081e12, rel=1e-3)
    assert bench.f_alg(28672, 8192) == pytest.approx(1.322e13, rel=1e-3)


def test_f_alg_small_cases_by_hand():
    # 1 x 2: one column split, E (1 x 1) times L^A_21 (1 x 1): 1 MAC
    assert bench.f_alg(1, 2) == 2.0
    # 2 x 1: one row split, L^B_21 (1 x 1) E (1 x 1): 1 MAC
    assert bench.f_alg(2, 1) == 2.0
    # 2 x 2: row split with L^B_21 E (1x1 @ 1x2: 2 MACs) and (.) L^A^T
    # (strictly-lower part of 2x2: 1 MAC per row, 1 row): 3 MACs, plus the two
    # 1 x 2 halves (1 MAC each)
    assert bench.f_alg(2, 2) == 2.0 * (3 + 1 + 1)
    # B = I: only the column splits' E L^A_21^T products remain: m n (n - 1) / 2
    for m, n in [(3, 5), (64, 64), (4096, 4096)]:
        assert bench.f_alg(m, n, identity_b=True) == m * n * (n - 1)


def test_fp32_effective_peak():
    p, src = bench.fp32_effective_peak({"bf16_tflops": 1892.3})
    assert p == pytest.approx(1892.3 / 6)
    assert "burst" in src


def test_top_left_block_sample_is_exact():
    """With the full problem's factors and per-row grid restricted to it, the
    top-left block solves to exactly the full solve's top-left codes."""
    W, A, B = WL.small_problem(96, 80, 17)
    W = W.numpy().astype(np.float64)
    f = O.prepare(A.numpy(), B.numpy(), 0.01)
    for group in (0, 16):
        full = O.bakron_recursive(W, f.LA, f.LB, O.quant_grid(W, 4, group))
        k = 48
        g = bench._grid_block(W, 4, group, k)
        blk = O.bakron_recursive(W[:k, :k], f.LA[:k, :k], f.LB[:k, :k], g, base=64)
        np.testing.assert_array_equal(blk.codes, full.codes[:k, :k])
        np.testing.assert_allclose(blk.X, full.X[:k, :k], atol=1e-10)


def test_traffic_is_per_launch_and_only_for_the_sources_it_was_taken_on(tmp_path, monkeypatch):
    """roofline.traffic: DRAM bytes per solve of a family from the committed
    summary, divided by the family's launches per solve; None for another
    workload, a family without a figure, or changed kernel sources."""
    import json
    import os
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.txt").write_text(json.dumps(
        {"csrc_hash": "abc", "workloads": {"config 2": {"leaf": 1000.0, "tc": 620.0}}}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "_csrc_hash", lambda: "abc")
    assert bench._traffic("config 2", "leaf", 250) == 4.0
    assert bench._traffic("config 2", "tc", 62) == 10.0
    assert bench._traffic("config 3", "tc", 62) is None
    assert bench._traffic("config 2", "simt", 10) is None
    assert bench._traffic("config 2", "tc", 0) is None
    monkeypatch.setattr(bench, "_csrc_hash", lambda: "changed")
    assert bench._traffic("config 2", "leaf", 250) is None
    assert os.path.exists(tmp_path / "profiles" / "traffic.txt")
