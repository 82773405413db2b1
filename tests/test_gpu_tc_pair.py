"""The band products on CTA pairs (BAKRON_TC_PAIR=1): two CTAs of a cluster
share one M = 256 tcgen05 MMA (cta_group::2), each holding its own 128 rows
of A and one half of B.  Checked: the diagnostic GEMM against fp64; the solve
with tensor-core bands forced down to width 2 (ragged shapes, odd numbers of
128-row blocks, so that pairs with one empty row block occur) against the
oracle; the same solves against the single-CTA kernel (each output entry is
the same sequence of MMAs, so the codes agree); the B = I column bands; the
bounded waits of the pair (a zero budget gives BAKRON_ERR_TIMEOUT for the
whole solve and leaves the context usable)."""
import numpy as np
import pytest
import torch

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


@pytest.fixture(autouse=True)
def _pairs(monkeypatch):
    monkeypatch.setenv("BAKRON_TC_PAIR", "1")
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    monkeypatch.setenv("BAKRON_LEAF_BLOCK", "4")


@pytest.mark.parametrize("M,N,K", [(256, 128, 32), (512, 384, 512), (768, 256, 1024)])
def test_pair_gemm_matches_fp64_and_single_cta(M, N, K, monkeypatch):
    g = torch.Generator(device="cuda").manual_seed(7 * M + N + K)
    A = torch.randn(M, K, device="cuda", generator=g)
    B = torch.randn(N, K, device="cuda", generator=g)
    C = P.bakron_diag_gemm_tf32x3(A, B).double()
    ref = A.double() @ B.double().T
    scale = A.double().abs() @ B.double().abs().T
    err = ((C - ref).abs() / scale).max().item()
    assert err < 2e-6, err
    monkeypatch.setenv("BAKRON_TC_PAIR", "0")
    C1 = P.bakron_diag_gemm_tf32x3(A, B).double()
    assert ((C - C1).abs() / scale).max().item() < 1e-6


@pytest.mark.parametrize("m,n", [(64, 64), (97, 131), (130, 300), (257, 129), (300, 417),
                                 (400, 350)])
def test_pair_solve_with_tensor_core_bands(m, n, monkeypatch):
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
    _assert_parity(_solve_small(m, n, 2000 + m + n, bits=4))


@pytest.mark.parametrize("group", [32, 128])
def test_pair_solve_groups(group, monkeypatch):
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "3")
    _assert_parity(_solve_small(150, 256, 33 + group, bits=3, group=group))


def test_pair_and_single_cta_agree(monkeypatch):
    """Same inputs through the paired and the single-CTA band kernels."""
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
    a = _solve_small(640, 520, 93, bits=4)
    monkeypatch.setenv("BAKRON_TC_PAIR", "0")
    b = _solve_small(640, 520, 93, bits=4)
    assert (a["codes"] == b["codes"]).all()
    S, _ = a["g"].expand(520)
    assert (np.abs(a["X"] - b["X"]) / S).max() < 1e-5


def test_pair_gptq_column_bands():
    """B = I: the column bands (MODE_COLS) on pairs against the general solve."""
    from tests.test_gpu_gptq import _gptq_small
    st, got, gp, X, S, W, fac = _gptq_small(290, 608, 4243, 4, 0)
    assert st["cert_mismatch_outside_band"] == 0, st
    general = P.bakron_solve(W.cuda(), fac, 4, 0)[0].cpu().numpy().astype(np.int64)
    assert (general == got).mean() == 1.0


def test_pair_bounded_waits_report_timeout_and_recover(monkeypatch):
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
    monkeypatch.setenv("BAKRON_SPIN_CYCLES", "0")
    with pytest.raises(P.BakronError) as e:
        _solve_small(300, 260, 5, bits=4)
    assert e.value.status == 4
    monkeypatch.delenv("BAKRON_SPIN_CYCLES")
    _assert_parity(_solve_small(300, 260, 5, bits=4))
