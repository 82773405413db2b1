"""Pins of the oracle's symmetric alphabet (Appendix "Experiments").

The paper's experiments round onto {-l, ..., +l} per row, with the scale set
to max |w| / l and then shrunk by up to a factor of 2 by an MSE search.  The
checks below compare ``symmetric_grid`` with hand-solved rows, invariants of
the definition, an independent error evaluation by enumeration of the
alphabet, and brute force of the whole solve over the finite alphabet.
"""
import numpy as np
import pytest

import oracle as O
import workloads as WL

F32 = np.float32


def _enumerated_errors(w, scales, levels):
    """Squared error of each value's nearest alphabet element, found by
    scanning all 2l+1 levels (no rint, no clamp)."""
    lv = np.arange(-levels, levels + 1, dtype=np.float64)
    out = []
    for s in np.asarray(scales, np.float64):
        d = (s * lv[None, :] - np.asarray(w, np.float64)[:, None]) ** 2
        out.append(d.min(axis=1).sum())
    return np.array(out)


def test_hand_solved_row():
    """l = 1, w = (1, 1/2, 1/2, 1/2), 8 shrink steps.  For s in (1/2, 1) the
    three halves round to s and the 1 clamps to s: error 3 (s - 1/2)^2 +
    (1 - s)^2, least at s = 5/8 (candidate k = 6: t = 10/16), value 3/16;
    the ends give 3/4 (s = 1) and 1/4 (s = 1/2)."""
    w = np.array([[1.0, 0.5, 0.5, 0.5]], F32)
    cand = O.symmetric_candidates(1.0, 1, 8)
    np.testing.assert_array_equal(cand, (16 - np.arange(9)) / 16.0)
    err = O.symmetric_errors(w[0], cand, 1)
    assert err[0] == pytest.approx(0.75, abs=1e-15)
    assert err[8] == pytest.approx(0.25, abs=1e-15)
    assert err[6] == pytest.approx(3 / 16, abs=1e-15)
    g = O.symmetric_grid(w, 1, shrink_steps=8)
    assert g.s[0, 0] == F32(0.625)
    assert g.z[0, 0] == 1 and g.qmax == 2
    r = O.rtn(w.astype(np.float64), g)
    np.testing.assert_array_equal(r.codes, [[2, 2, 2, 2]])   # all at +s


def test_lattice_row_keeps_full_scale():
    """A row already on the lattice of max|w| / l is reproduced (almost)
    exactly at k = 0, and every shrink clamps its largest entry."""
    levels = 3
    w = (np.array([3, -2, 1, 0, -3, 2], np.float64) * 0.5).astype(F32)
    g = O.symmetric_grid(w[None, :], levels, shrink_steps=50)
    cand = O.symmetric_candidates(1.5, levels, 50)
    assert g.s[0, 0] == cand[0]
    assert O.symmetric_errors(w, cand[:1], levels)[0] < 1e-12


def test_candidates_span_half_to_full():
    """K + 1 strictly decreasing scales from max|w|/l down to max|w|/(2l)."""
    for amax, levels, K in [(0.37, 3, 50), (2.0, 1, 10), (1e-3, 7, 64)]:
        c = O.symmetric_candidates(amax, levels, K).astype(np.float64)
        assert len(c) == K + 1
        assert np.all(np.diff(c) < 0)
        assert c[0] == pytest.approx(amax / levels, rel=2e-7)
        assert c[-1] == pytest.approx(amax / (2 * levels), rel=2e-7)
    # K = 0: the plain max-abs scale, exact for l = 1
    assert O.symmetric_candidates(0.75, 1, 0)[0] == F32(0.75)
    np.testing.assert_array_equal(O.symmetric_candidates(0.75, 3, 0),
                                  [F32(np.float64(F32(0.75)) * np.float64(F32(1 / 3)))])


def test_errors_match_enumeration():
    """rint + clamp gives the nearest alphabet element: the error equals the
    one found by scanning the alphabet."""
    rng = np.random.default_rng(5)
    for levels in (1, 3, 7):
        w = rng.standard_t(4, size=200).astype(F32)
        cand = O.symmetric_candidates(np.abs(w).max(), levels, 50)
        np.testing.assert_allclose(O.symmetric_errors(w, cand, levels),
                                   _enumerated_errors(w, cand, levels), rtol=1e-12)


def test_grid_is_the_least_error_candidate():
    rng = np.random.default_rng(11)
    W = rng.standard_t(5, size=(24, 96)).astype(F32)
    for group in (0, 32):
        g = O.symmetric_grid(W, 3, group=group, shrink_steps=50)
        gs = 96 if group == 0 else group
        for i in range(24):
            for j in range(96 // gs):
                w = W[i, j * gs:(j + 1) * gs]
                cand = O.symmetric_candidates(np.abs(w).max(), 3, 50)
                err = _enumerated_errors(w, cand, 3)
                k = int(np.flatnonzero(cand == g.s[i, j])[0])
                assert err[k] <= err.min() * (1 + 1e-12)
                assert np.all(err[:k] > err[k] * (1 - 1e-12) - 1e-300) or k == 0
        assert np.all(g.z == 3) and g.qmax == 6


def test_symmetry_and_scaling():
    """Negating a row leaves the grid unchanged; scaling it by 2^e scales the
    scale by 2^e exactly; an all-zero row uses max|w| = 1."""
    rng = np.random.default_rng(3)
    W = rng.normal(size=(10, 64)).astype(F32)
    g = O.symmetric_grid(W, 3)
    np.testing.assert_array_equal(O.symmetric_grid(-W, 3).s, g.s)
    np.testing.assert_array_equal(O.symmetric_grid(W * F32(4), 3).s, g.s * F32(4))
    np.testing.assert_array_equal(O.symmetric_grid(W * F32(0.125), 3).s, g.s * F32(0.125))
    Z = np.zeros((2, 8), F32)
    gz = O.symmetric_grid(Z, 3)
    np.testing.assert_array_equal(gz.s, np.full((2, 1), O.symmetric_candidates(1, 3, 50)[0]))


def test_mse_search_never_worse_than_max_abs():
    rng = np.random.default_rng(8)
    W = rng.standard_t(3, size=(40, 128)).astype(F32)
    g = O.symmetric_grid(W, 3)
    g0 = O.symmetric_grid(W, 3, shrink_steps=0)
    e = O.rtn(W.astype(np.float64), g).V - W
    e0 = O.rtn(W.astype(np.float64), g0).V - W
    assert np.all((e ** 2).sum(1) <= (e0 ** 2).sum(1) * (1 + 1e-12))
    assert (e ** 2).sum() < (e0 ** 2).sum()   # heavy tails: shrinking pays


@pytest.mark.parametrize("m,n", [(1, 4), (2, 3), (3, 2), (2, 2)])
def test_brute_force_with_symmetric_alphabet(m, n):
    """Over {-1, 0, 1}^{mn} exactly one V is a fixed point of the
    certificate; it is every tier's output; the CVP minimum is below it."""
    W, A, B = WL.small_problem(m, n, 700 + 10 * m + n)
    W = W.numpy().astype(np.float64)
    f = O.prepare(A.numpy(), B.numpy(), 0.01)
    g = O.symmetric_grid(W.astype(F32), 1, shrink_steps=8)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    for solver in (O.bakron_naive, O.bakron_recursive, O.bakron):
        np.testing.assert_array_equal(solver(W, f.LA, f.LB, g).codes, ref.codes)
    fixed, best = O.brute_force(W, f.LA, f.LB, f.A_d, f.B_d, g)
    assert len(fixed) == 1
    np.testing.assert_array_equal(fixed[0], ref.codes)
    assert best <= O.objective(W, ref.V, f.A_d, f.B_d) + 1e-15


def test_solve_with_symmetric_grid_beats_rtn():
    W, A, B = WL.small_problem(48, 40, 77)
    W = W.numpy().astype(np.float64)
    f = O.prepare(A.numpy(), B.numpy(), 0.5)     # the paper's damping for its runs
    g = O.symmetric_grid(W.astype(F32), 3)
    r = O.bakron(W, f.LA, f.LB, g)
    rt = O.rtn(W, g)
    assert O.objective(W, r.V, f.A_d, f.B_d) < O.objective(W, rt.V, f.A_d, f.B_d)
    assert r.codes.min() >= 0 and r.codes.max() <= 6


def test_planted_quantiser_mistakes_are_caught():
    """Slips in copies of the search change the hand-solved row's answer."""
    w = np.array([1.0, 0.5, 0.5, 0.5])
    cand = O.symmetric_candidates(1.0, 1, 8).astype(np.float64)
    good = cand[int(np.argmin(O.symmetric_errors(w, cand, 1)))]
    # no clamp: the 1 rounds to 2s, and s = 1/2 becomes exact
    no_clamp = (((cand[:, None] * np.rint(w[None, :] / cand[:, None])) - w) ** 2).sum(1)
    assert cand[int(np.argmin(no_clamp))] != good
    # shrink applied as a division (scales above max|w|/l)
    up = 1.0 / cand * cand[0] ** 2
    assert up.max() == pytest.approx(2 * cand[0]) and up.min() == cand[0]
    assert up[int(np.argmin(O.symmetric_errors(w, up, 1)))] != good
    # asymmetric clamp to [-l, l-1]
    asym = ((cand[:, None] * np.clip(np.rint(w[None, :] / cand[:, None]), -1, 0) - w) ** 2).sum(1)
    assert cand[int(np.argmin(asym))] != good
