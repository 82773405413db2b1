"""Persistent cooperative launches of the narrow ranges of the recursion
(leaves and band products of rec(k, l) for l - k <= BAKRON_SUBTREE_MAX, as
phases separated by grid-wide barriers) against the oracle, against the
launch-per-kernel path, and the bounded barrier wait."""
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
def _small_leaf_blocks(monkeypatch):
    """Blocks of at most 4 leaves, so that these small problems still have
    band nodes of every width (the default blocks of 8 leave none below 9)."""
    monkeypatch.setenv("BAKRON_LEAF_BLOCK", "4")


@pytest.mark.parametrize("width", ["2", "3", "8", "16", "32"])
@pytest.mark.parametrize("m,n", [(97, 131), (300, 417), (640, 96)])
def test_subtree_widths(width, m, n, monkeypatch):
    """Every range width up to the widest, on ragged shapes (partial tiles,
    more tiles on a diagonal than one CTA, tall and wide)."""
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", width)
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    _assert_parity(_solve_small(m, n, 7000 + m + n, bits=4))


@pytest.mark.parametrize("fused", ["0", "4", "64"])
def test_subtree_band_forms(fused, monkeypatch):
    """Inside a subtree, bands run fused or as two stages."""
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "32")
    monkeypatch.setenv("BAKRON_FUSED_MAX_BAND", fused)
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    _assert_parity(_solve_small(250, 330, 77, bits=3))


def test_subtree_with_tensor_core_bands_above(monkeypatch):
    """Subtrees below, tensor-core bands above them."""
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "4")
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "5")
    _assert_parity(_solve_small(500, 380, 31, bits=4, group=0))


def test_subtree_matches_launch_per_kernel(monkeypatch):
    """Same arithmetic per tile and per band unit, so the codes agree with the
    launch-per-kernel path exactly and the pre-rounding values bit for bit."""
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    a = _solve_small(420, 380, 12, bits=4)
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "8")
    b = _solve_small(420, 380, 12, bits=4)
    assert np.array_equal(a["codes"], b["codes"])
    assert np.array_equal(a["X"], b["X"])


def test_subtree_barrier_timeout_and_recover(monkeypatch):
    """A zero wait budget makes the grid barrier's waits run out (several CTAs
    per phase): BAKRON_ERR_TIMEOUT, no hang, and the next solve is correct."""
    monkeypatch.setenv("BAKRON_TC_MIN_BAND", "0")
    monkeypatch.setenv("BAKRON_SUBTREE_MAX", "32")
    monkeypatch.setenv("BAKRON_SPIN_CYCLES", "0")
    # 19 x 14 tiles, 32 tile anti-diagonals: one subtree of two leaf blocks
    # and the band between them, up to 14 CTAs per phase
    with pytest.raises(P.BakronError) as e:
        _solve_small(600, 420, 5, bits=4)
    assert e.value.status == 4
    monkeypatch.delenv("BAKRON_SPIN_CYCLES")
    _assert_parity(_solve_small(600, 420, 5, bits=4))
