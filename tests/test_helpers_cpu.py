"""CPU checks of the test helpers the GPU parity tests rely on."""
import numpy as np

from tests._helpers import root_mismatches


def test_root_mismatches_hand_case():
    bad = np.zeros((5, 6), bool)
    bad[1, 3] = bad[2, 4] = bad[3, 1] = bad[4, 0] = True
    r = root_mismatches(bad)
    # (2, 4) lies below-right of (1, 3); (4, 0) is left of (3, 1), not below-right
    want = bad.copy()
    want[2, 4] = False
    np.testing.assert_array_equal(r, want)


def test_root_mismatches_brute_force():
    rng = np.random.default_rng(3)
    for _ in range(20):
        bad = rng.random((7, 9)) < 0.15
        r = root_mismatches(bad)
        for p in range(7):
            for q in range(9):
                cone = bad[:p + 1, :q + 1].copy()
                cone[p, q] = False
                assert r[p, q] == (bad[p, q] and not cone.any())
