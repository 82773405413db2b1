"""bakron_autotune: it picks a candidate schedule, later solves of that shape
use it (and still give the oracle's codes), the environment overrides it,
and clearing the table restores the defaults."""
import os

import pytest
import torch

import workloads as WL
from tests._helpers import oracle_factors_fp32
from tests.test_gpu_parity import _assert_parity, _solve_small

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    P.lib()
    yield
    P.bakron_autotune_clear()


def _problem(m, n, seed):
    W, A, B = WL.small_problem(m, n, seed)
    f, LA32, LB32 = oracle_factors_fp32(A, B, 0.01)
    dev = "cuda"
    fac = P.bakron_set_factors(torch.from_numpy(LA32).to(dev), torch.from_numpy(LB32).to(dev),
                               None, None)
    return W.to(dev), fac


def test_autotune_choice_is_used_and_cleared(monkeypatch):
    for v in ("BAKRON_TC_MIN_BAND", "BAKRON_FUSED_MAX_BAND", "BAKRON_LEAF_BLOCK"):
        monkeypatch.delenv(v, raising=False)
    P.bakron_autotune_clear()
    m, n = 520, 610
    default = {"tc_min_band": 6, "fused_max_band": 2, "leaf_block": 8}
    assert P.bakron_get_tuning(m, n) == default
    W, fac = _problem(m, n, 3)
    best = P.bakron_autotune(W, fac, 4, 0)
    assert best["tc_min_band"] in (0, 4, 6, 8, 12, 16, 24)
    assert best["fused_max_band"] in (2, 4)
    assert best["leaf_block"] in (4, 8, 16)
    assert best["ms"] > 0
    got = P.bakron_get_tuning(m, n)
    assert got == {k: best[k] for k in ("tc_min_band", "fused_max_band", "leaf_block")}
    # a solve of the tuned shape launches what the same thresholds set by hand launch
    P.bakron_solve(W, fac, 4, 0)
    tuned_launches = P.bakron_last_launches()
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", str(best["tc_min_band"]))
    monkeypatch.setenv("BAKRON_FUSED_MAX_BAND", str(best["fused_max_band"]))
    monkeypatch.setenv("BAKRON_LEAF_BLOCK", str(best["leaf_block"]))
    P.bakron_solve(W, fac, 4, 0)
    assert P.bakron_last_launches() == tuned_launches
    # the environment wins over the table
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    assert P.bakron_get_tuning(m, n)["tc_min_band"] == 0
    monkeypatch.delenv("BAKRON_TC_MIN_BAND")
    monkeypatch.delenv("BAKRON_FUSED_MAX_BAND")
    monkeypatch.delenv("BAKRON_LEAF_BLOCK")
    P.bakron_autotune_clear()
    assert P.bakron_get_tuning(m, n) == default


def test_tuned_solve_keeps_parity(monkeypatch):
    for v in ("BAKRON_TC_MIN_BAND", "BAKRON_FUSED_MAX_BAND", "BAKRON_LEAF_BLOCK"):
        monkeypatch.delenv(v, raising=False)
    m, n = 300, 417
    W, fac = _problem(m, n, 2000 + m + n)
    P.bakron_autotune(W, fac, 4, 0)
    _assert_parity(_solve_small(m, n, 2000 + m + n, bits=4))
    P.bakron_autotune_clear()
