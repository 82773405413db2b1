"""The tcgen05 3xTF32 band products: the diagnostic GEMM against fp64, and the
solve with the tensor-core path forced onto every band of width >= 2 (so that
small, ragged problems exercise the band masks) against the oracle.  These
tests turn the persistent subtree launches off (BAKRON_SUBTREE_MAX=0), which
would otherwise take every narrow band of a small problem."""
import numpy as np
import pytest
import torch

import oracle as O
from tests._helpers import compare_codes
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
def _small_leaf_blocks(monkeypatch):
    """Blocks of at most 4 leaves, so that these small problems still have
    band nodes of every width (the default blocks of 8 leave none below 9)."""
    monkeypatch.setenv("BAKRON_LEAF_BLOCK", "4")


@pytest.mark.parametrize("M,N,K", [(128, 128, 32), (256, 384, 512), (384, 128, 1024)])
def test_gemm_3xtf32_matches_fp64(M, N, K):
    g = torch.Generator(device="cuda").manual_seed(M + N + K)
    A = torch.randn(M, K, device="cuda", generator=g)
    B = torch.randn(N, K, device="cuda", generator=g)
    C = P.bakron_diag_gemm_tf32x3(A, B).double()
    ref = A.double() @ B.double().T
    scale = A.double().abs() @ B.double().abs().T
    err = ((C - ref).abs() / scale).max().item()
    assert err < 2e-6, err          # fp32-class; 1xTF32 would be ~1e-3


def test_gemm_3xtf32_structured_zeros():
    """Triangular operands (as the factors are) give exact zeros where a row of
    A and a row of B have disjoint support."""
    A = torch.tril(torch.randn(256, 256, device="cuda"))
    B = torch.eye(256, device="cuda")
    C = P.bakron_diag_gemm_tf32x3(A, B)
    assert torch.equal(C.triu(1), torch.zeros_like(C).triu(1))
    assert ((C - A).abs().max() / A.abs().max()).item() < 1e-6


@pytest.mark.parametrize("m,n", [(64, 64), (97, 131), (130, 300), (257, 129), (300, 417)])
def test_solve_with_tensor_core_bands(m, n, monkeypatch):
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
    _assert_parity(_solve_small(m, n, 2000 + m + n, bits=4))


@pytest.mark.parametrize("group", [32, 128])
def test_solve_with_tensor_core_bands_groups(group, monkeypatch):
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "3")
    _assert_parity(_solve_small(150, 256, 33 + group, bits=3, group=group))


def test_tensor_core_and_simt_paths_agree(monkeypatch):
    """Same inputs, band products on tcgen05 vs on CUDA cores: identical codes
    (the difference is ~1e-6 of an update, far inside the tie band)."""
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    a = _solve_small(400, 350, 91, bits=4)
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
    b = _solve_small(400, 350, 91, bits=4)
    assert (a["codes"] == b["codes"]).mean() >= 0.999
    S, _ = a["g"].expand(350)
    assert (np.abs(a["X"] - b["X"]) / S)[a["codes"] == b["codes"]].max() < 1e-4


def test_bounded_waits_report_timeout_and_recover(monkeypatch):
    """A zero wait budget makes the tensor-core waits run out: the solve returns
    BAKRON_ERR_TIMEOUT (no hang, no fault) and the next solve is correct."""
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
    monkeypatch.setenv("BAKRON_SPIN_CYCLES", "0")
    with pytest.raises(P.BakronError) as e:
        _solve_small(200, 260, 5, bits=4)
    assert e.value.status == 4
    monkeypatch.delenv("BAKRON_SPIN_CYCLES")
    _assert_parity(_solve_small(200, 260, 5, bits=4))


@pytest.mark.parametrize("fused", ["0", "4", "64"])
def test_solve_with_fused_narrow_bands(fused, monkeypatch):
    """Narrow Alg. 5 nodes with both stages fused in one launch (all widths up
    to 64 when forced) give the oracle's codes."""
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    monkeypatch.setenv("BAKRON_FUSED_MAX_BAND", fused)
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    _assert_parity(_solve_small(160, 230, 404, bits=4))


def test_mma_rate_diagnostic():
    """The measured tcgen05 kind::tf32 rate is a plausible whole-GPU figure
    (GB300 nominal dense tf32: 1.1 PFLOP/s; one MMA of 128 x 128 x 8 per SM
    takes at least 32 cycles)."""
    r = P.bakron_diag_mma_rate(500)
    assert 100.0 < r["tf32_tflops"] < 3000.0, r
    assert r["cycles_per_mma"] >= 32.0, r
