"""Pins of the float64 oracle against facts the paper and the mathematics fix.

Every check here compares the oracle with something other than itself: a
hand-worked example, a textbook algorithm written from its own paper, closed
forms, invariants, special cases, brute force, and the equivalence theorem's
cross-tier equality (Thm. 3.1).  A plausible slip in the oracle (a dropped
term, a wrong sign or index, a transposed factor, the "original W" misreading
of Alg. 4/5) fails at least one of them; ``test_planted_mistakes_are_caught``
shows this for a few such slips.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _problem(m, n, seed, bits=None, group=0, damp=0.01):
    W, A, B = WL.small_problem(m, n, seed)
    W = W.numpy().astype(np.float64)
    f = O.prepare(A.numpy(), B.numpy(), damp)
    g = O.integer_grid(m) if bits is None else O.quant_grid(W, bits, group)
    if bits is None:
        W = W * 50.0  # spread over several integers so rounding is non-trivial
    return W, f, g


# --------------------------------------------------------------------- golden
def test_hand_worked_2x2():
    """Alg. 2 worked by hand on a 2x2 problem (tests/golden/hand_2x2.json)."""
    gd = json.load(open(os.path.join(GOLDEN, "hand_2x2.json")))
    W, A, B = (np.array(gd[k]) for k in ("W", "A", "B"))
    f = O.prepare(A, B, damp=0.0)
    np.testing.assert_allclose(f.LA, gd["LA"], atol=1e-14)
    np.testing.assert_allclose(f.LB, gd["LB"], atol=1e-14)
    np.testing.assert_allclose(f.rA, gd["rA"], rtol=1e-14)
    np.testing.assert_allclose(f.rB, gd["rB"], rtol=1e-14)
    g = O.integer_grid(2)
    for solver in (O.bakron_naive, O.bakron_antidiagonal, O.bakron_recursive, O.bakron):
        r = solver(W, f.LA, f.LB, g)
        np.testing.assert_array_equal(r.codes, gd["V"])
        np.testing.assert_allclose(r.X, gd["X"], atol=1e-14)
    r = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    np.testing.assert_array_equal(r.codes, gd["V"])
    np.testing.assert_allclose(r.X, gd["X"], atol=1e-14)
    assert O.objective(W, r.V, f.A_d, f.B_d) == pytest.approx(gd["objective"], rel=1e-13)
    assert O.objective_from_errors(r.E, f.rA, f.rB) == pytest.approx(gd["objective"], rel=1e-13)
    rt = O.rtn(W, g)
    np.testing.assert_array_equal(rt.codes, gd["rtn_V"])
    assert O.objective(W, rt.V, f.A_d, f.B_d) == pytest.approx(gd["rtn_objective"], rel=1e-13)


# ------------------------------------------------------------------ quantiser
def test_grid_hand_cases():
    """Asymmetric min-max grid on exactly representable values."""
    W = np.array([[-0.75, 0.2, 0.75, 0.0],
                  [0.5, 1.5, 0.25, 3.0]])
    g = O.quant_grid(W, 2)
    # row 0: range [-0.75, 0.75], s = 0.5, z = rint(1.5) = 2 (half to even)
    assert g.s[0, 0] == np.float32(0.5) and g.z[0, 0] == 2
    # row 1: range [0, 3] (0 is included), s = 1, z = 0
    assert g.s[1, 0] == np.float32(1.0) and g.z[1, 0] == 0
    c, v = O.quantize(W[0], 0.5, 2, 3)
    np.testing.assert_array_equal(c, [0, 2, 3, 2])   # 0.75/0.5 = 1.5 -> 2 -> clamp 3
    np.testing.assert_array_equal(v, [-1.0, 0.0, 0.5, 0.0])
    # ties go to the even integer of x/s
    c, _ = O.quantize(np.array([0.25, 0.75, -0.25]), 0.5, 2, 3)
    np.testing.assert_array_equal(c, [2, 3, 2])  # x/s: 0.5->0, 1.5->2 (clamped), -0.5->0
    # groups of two columns get their own range
    gg = O.quant_grid(W, 2, group=2)
    assert gg.s.shape == (2, 2)
    assert gg.s[1, 1] == np.float32(1.0) and gg.z[1, 1] == 0      # [0.25, 3] -> [0, 3]
    assert gg.s[0, 1] == np.float32(0.25) and gg.z[0, 1] == 0     # [0, 0.75]


def test_grid_degenerate_row_and_group_errors():
    W = np.zeros((1, 4))
    g = O.quant_grid(W, 3)
    assert g.s[0, 0] > 0
    c, v = O.quantize(0.0, g.s[0, 0], g.z[0, 0], g.qmax)
    assert v == 0.0                      # zero is on the grid
    with pytest.raises(ValueError):
        O.quant_grid(np.zeros((2, 6)), 2, group=4)


def test_midpoint_distance_hand_values():
    """Distance in grid units from x/s to the nearest rounding boundary (a
    half-integer), which decides what the certificate excuses as a tie.
    Hand values: on a boundary 0, on an integer 1/2, just below a boundary the
    gap, and negative values measured to the boundary on their own side."""
    d = O.midpoint_distance
    assert d(2.5, 1.0) == 0.0
    assert d(-2.5, 1.0) == 0.0
    assert d(3.0, 1.0) == 0.5
    assert d(-3.0, 1.0) == 0.5
    assert d(0.0, 1.0) == 0.5
    assert d(4.49999, 1.0) == pytest.approx(1e-5, abs=1e-12)
    assert d(4.50001, 1.0) == pytest.approx(1e-5, abs=1e-12)
    assert d(-0.3, 1.0) == pytest.approx(0.2, abs=1e-12)       # nearest boundary -0.5
    assert d(-0.7, 1.0) == pytest.approx(0.2, abs=1e-12)       # nearest boundary -0.5
    assert d(1.2, 1.0) == pytest.approx(0.3, abs=1e-12)        # nearest boundary 1.5
    # grid units: x = 0.75 on a grid of step 0.5 is 1.5 units, on a boundary
    assert d(0.75, 0.5) == 0.0
    assert d(0.5, 0.5) == 0.5
    assert d(-0.2, 0.5) == pytest.approx(0.1, abs=1e-12)       # -0.4 units
    # a tie exactly at the boundary is where rint's half-to-even rule acts
    x = np.array([0.5, 1.5, 2.5, -0.5])
    assert (O.midpoint_distance(x, 1.0) == 0).all()
    np.testing.assert_array_equal(np.rint(x), [0.0, 2.0, 2.0, -0.0])


def test_babai_step_is_argmin_over_alphabet():
    """Babai's greedy step picks the nearest alphabet element (P1)."""
    rng = np.random.default_rng(5)
    for _ in range(400):
        s = float(rng.uniform(0.01, 1.0))
        z = float(rng.integers(0, 8))
        x = float(rng.normal(0.0, 4.0 * s))
        c, _ = O.quantize(x, s, z, 7)
        assert int(c) == O.babai_step_by_enumeration(x, s, z, 7)


# -------------------------------------------------------------------- factors
def test_kronecker_vec_identity():
    """Prop. 3.1 with column-major vec: (A (x) B) vec(W) = vec(B W A^T)."""
    rng = np.random.default_rng(1)
    A, B, W = rng.normal(size=(4, 4)), rng.normal(size=(3, 3)), rng.normal(size=(3, 4))
    lhs = np.kron(A, B) @ W.reshape(-1, order="F")
    np.testing.assert_allclose(lhs, (B @ W @ A.T).reshape(-1, order="F"), atol=1e-12)


@pytest.mark.parametrize("d", [1, 2, 7, 40])
def test_factor_definitions_agree(d):
    """Cholesky(H^-1) normalised == RevCholesky(H)^-1 diag(R), and R^T R = H."""
    _, A, _ = WL.small_problem(2, d, 11)
    H = O.damped(A.numpy(), 0.01)
    R = O.rev_cholesky(H)
    assert np.allclose(np.triu(R, 1), 0) and (np.diag(R) > 0).all()
    np.testing.assert_allclose(R.T @ R, H, rtol=1e-12, atol=1e-14 * np.abs(H).max())
    L1, L2 = O.unit_lower_factor(H), O.unit_lower_factor_via_rev(H)
    np.testing.assert_allclose(np.diag(L1), 1.0, atol=1e-14)
    np.testing.assert_allclose(L1, L2, atol=1e-9 * max(1.0, np.abs(L1).max()))
    # L^-1 = diag(R)^-1 R : the identity the certificate relies on
    np.testing.assert_allclose(np.linalg.inv(L1), R / np.diag(R)[:, None], atol=1e-8)


def test_damping():
    H = np.array([[2.0, 0.5], [0.5, 4.0]])
    np.testing.assert_allclose(O.damped(H, 0.1), H + 0.3 * np.eye(2))


# --------------------------------------------------------------- cross tiers
SHAPES = [(1, 1), (1, 6), (6, 1), (3, 5), (5, 3), (6, 6), (7, 4), (2, 9)]


@pytest.mark.parametrize("m,n", SHAPES)
@pytest.mark.parametrize("bits", [None, 2, 4])
def test_all_tiers_agree(m, n, bits):
    """Thm. 3.1: Alg. 2, 3, 4, 5 and the explicit vectorised definition give
    the same codes (and the same pre-rounding workspace)."""
    W, f, g = _problem(m, n, 100 + 7 * m + n, bits)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    for solver in (O.bakron_naive, O.bakron_antidiagonal, O.bakron_recursive, O.bakron):
        r = solver(W, f.LA, f.LB, g)
        np.testing.assert_array_equal(r.codes, ref.codes)
        np.testing.assert_allclose(r.X, ref.X, atol=1e-10)


@pytest.mark.parametrize("m,n", [(1, 7), (7, 1), (5, 9), (9, 5), (13, 11), (16, 16)])
@pytest.mark.parametrize("base", [2, 3, 4, 8])
def test_blocked_recursive_agrees(m, n, base):
    """Alg. 4 stopped at blocks of at most base x base, each rounded by Alg. 3
    restricted to the block, gives the definition's codes and pre-rounding
    workspace (Thm. 3.1), also where blocks are ragged."""
    W, f, g = _problem(m, n, 500 + 3 * m + n + base, bits=3)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    r = O.bakron_recursive(W, f.LA, f.LB, g, base=base)
    np.testing.assert_array_equal(r.codes, ref.codes)
    np.testing.assert_allclose(r.X, ref.X, atol=1e-10)
    np.testing.assert_allclose(r.V, ref.V, atol=1e-12)


def test_blocked_recursive_agrees_medium_with_groups():
    """The blocked tier at the block sizes the full-size comparisons use, on a
    problem several blocks wide with a ragged tail and column groups."""
    W, f, g = _problem(150, 136, 41, bits=4, group=8)
    ref = O.bakron_recursive(W, f.LA, f.LB, g)
    for base in (32, 64):
        r = O.bakron_recursive(W, f.LA, f.LB, g, base=base)
        np.testing.assert_array_equal(r.codes, ref.codes)
        np.testing.assert_allclose(r.X, ref.X, atol=1e-10)


def test_tiers_agree_with_groups():
    W, f, g = _problem(5, 8, 77, bits=3, group=4)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    for solver in (O.bakron_naive, O.bakron_recursive, O.bakron):
        np.testing.assert_array_equal(solver(W, f.LA, f.LB, g).codes, ref.codes)


def test_recursive_and_band_agree_medium():
    """Alg. 4 and Alg. 5 on a 48 x 40 problem with a 4-bit grid."""
    W, f, g = _problem(48, 40, 5, bits=4)
    a = O.bakron_recursive(W, f.LA, f.LB, g)
    b = O.bakron(W, f.LA, f.LB, g)
    np.testing.assert_array_equal(a.codes, b.codes)
    np.testing.assert_allclose(a.X, b.X, atol=1e-10)


# ---------------------------------------------------------------- brute force
@pytest.mark.parametrize("m,n", [(1, 3), (2, 2), (2, 3), (3, 2)])
def test_brute_force_unique_fixed_point(m, n):
    """Over the whole alphabet^{mn} exactly one V satisfies V = Q(X(V)), it is
    the oracle's output, and the exhaustive CVP minimum is below it."""
    W, f, g = _problem(m, n, 300 + m * 10 + n, bits=2)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    fixed, best = O.brute_force(W, f.LA, f.LB, f.A_d, f.B_d, g)
    assert len(fixed) == 1
    np.testing.assert_array_equal(fixed[0], ref.codes)
    assert best <= O.objective(W, ref.V, f.A_d, f.B_d) + 1e-15


# --------------------------------------------------------------- certificate
def test_certificate_accepts_output_and_rejects_flip():
    W, f, g = _problem(12, 9, 8, bits=3)
    r = O.bakron_recursive(W, f.LA, f.LB, g)
    X, bad, _ = O.certificate(W, r.codes, g, f.LA, f.LB)
    assert not bad.any()
    np.testing.assert_allclose(X, r.X, atol=1e-10)
    # flip one code: its own pre-rounding value does not move, so the
    # certificate must fail exactly there (and nowhere before it)
    codes = r.codes.copy()
    p, q = 5, 4
    codes[p, q] = codes[p, q] + 1 if codes[p, q] < g.qmax else codes[p, q] - 1
    _, bad, _ = O.certificate(W, codes, g, f.LA, f.LB)
    assert bad[p, q]
    K = np.add.outer(np.arange(12), np.arange(9))
    assert not bad[K < p + q].any()


# ------------------------------------------------------------------ objective
def test_objective_identity_and_bound():
    """P3: tr((W-V)^T B (W-V) A) = sum (E rB rA)^2.  Cor. 3.3 bound on Z."""
    W, f, g = _problem(14, 11, 21, bits=None)
    r = O.bakron(W, f.LA, f.LB, g)
    obj = O.objective(W, r.V, f.A_d, f.B_d)
    assert obj == pytest.approx(O.objective_from_errors(r.E, f.rA, f.rB), rel=1e-10)
    assert np.abs(r.E).max() <= 0.5 + 1e-12
    bound = O.error_bound(g, f.rA, f.rB, W.shape[1])
    assert obj <= bound
    assert bound <= 0.25 * np.trace(f.A_d) * np.trace(f.B_d) * (1 + 1e-12)


@pytest.mark.parametrize("seed", range(6))
def test_beats_round_to_nearest(seed):
    """Expected (not a theorem): error feedback lowers the objective vs RTN."""
    W, f, g = _problem(24, 20, 500 + seed, bits=3)
    r = O.bakron_recursive(W, f.LA, f.LB, g)
    t = O.rtn(W, g)
    assert O.objective(W, r.V, f.A_d, f.B_d) < O.objective(W, t.V, f.A_d, f.B_d)


# -------------------------------------------------------------- special cases
def test_b_identity_is_gptq():
    """B = I: the solve is per-row GPTQ with H = A (Sec. 1), checked against the
    textbook GPTQ loop (upper Cholesky of H^-1, error / U_ii)."""
    W, f, g = _problem(6, 10, 41, bits=3)
    LB = O.unit_lower_factor(O.damped(np.eye(6), 0.01))
    np.testing.assert_allclose(LB, np.eye(6), atol=1e-15)
    r = O.bakron_recursive(W, f.LA, LB, g)
    S, Z = g.expand(10)
    gp = O.gptq_rows(W, f.A_d, S, Z, g.qmax)
    np.testing.assert_array_equal(r.codes, gp.codes)


def test_a_identity_is_column_gptq():
    """A = I: each column is GPTQ under H = B with the per-row grid."""
    W, f, g = _problem(9, 5, 42, bits=3)
    r = O.bakron(W, np.eye(5), f.LB, g)
    S, Z = g.expand(5)
    gp = O.gptq_rows(W.T, f.B_d, S.T, Z.T, g.qmax)
    np.testing.assert_array_equal(r.codes, gp.codes.T)


def test_diagonal_factors_are_rtn():
    W, _, g = _problem(7, 6, 43, bits=4)
    A = np.diag(np.linspace(1, 3, 6))
    B = np.diag(np.linspace(2, 5, 7))
    f = O.prepare(A, B, 0.01)
    np.testing.assert_allclose(f.LA, np.eye(6), atol=1e-15)
    np.testing.assert_array_equal(O.bakron(W, f.LA, f.LB, g).codes, O.rtn(W, g).codes)


# ------------------------------------------------------------------ configs
def test_config1_recursive_equals_band():
    """Config 1 (128 x 128, 4-bit per row): Alg. 4 == Alg. 5 and beats RTN."""
    W, A, B = WL.make(1)
    W = W.numpy().astype(np.float64)
    f = O.prepare(A.numpy(), B.numpy(), 0.01, via_inverse=False)
    g = O.quant_grid(W, 4)
    a = O.bakron_recursive(W, f.LA, f.LB, g)
    b = O.bakron(W, f.LA, f.LB, g)
    np.testing.assert_array_equal(a.codes, b.codes)
    _, bad, _ = O.certificate(W, a.codes, g, f.LA, f.LB)
    assert not bad.any()
    assert O.objective(W, a.V, f.A_d, f.B_d) < O.objective(W, O.rtn(W, g).V, f.A_d, f.B_d)


# ------------------------------------------------------ quadrant recursion
def _quadrant_order(W, LA, LB, grid):
    """The rounding in another order than every tier of the oracle: recursion
    over quadrants, top-left first, then top-right and bottom-left (no entry
    of either precedes one of the other), then bottom-right; after each
    quadrant its errors are added to the quadrants after it in the block.
    Written here, apart from the oracle, from the dependency structure of
    Sec. 3.3 (an entry's error reaches only entries below and right of it)."""
    X = np.asarray(W, np.float64).copy()
    m, n = X.shape
    S, Z = grid.expand(n)
    codes = np.zeros((m, n), np.int64)
    E = np.zeros((m, n))

    def spread(r0, r1, c0, c1, targets):
        Eb = np.zeros((m, n))
        Eb[r0:r1, c0:c1] = E[r0:r1, c0:c1]
        upd = LB @ Eb @ LA.T
        for (a0, a1, b0, b1) in targets:
            X[a0:a1, b0:b1] += upd[a0:a1, b0:b1]

    def rec(r0, r1, c0, c1):
        if r1 - r0 == 1 and c1 - c0 == 1:
            c, v = O.quantize(X[r0, c0], S[r0, c0], Z[r0, c0], grid.qmax)
            codes[r0, c0] = int(c)
            E[r0, c0] = v - X[r0, c0]
            return
        rm = (r0 + r1) // 2 if r1 - r0 > 1 else r1
        cm = (c0 + c1) // 2 if c1 - c0 > 1 else c1
        tl, tr, bl, br = (r0, rm, c0, cm), (r0, rm, cm, c1), (rm, r1, c0, cm), (rm, r1, cm, c1)
        live = lambda b: b[0] < b[1] and b[2] < b[3]
        rec(*tl)
        spread(*tl, [b for b in (tr, bl, br) if live(b)])
        for b in (tr, bl):
            if live(b):
                rec(*b)
                if live(br):
                    spread(*b, [br])
        if live(br):
            rec(*br)

    rec(0, m, 0, n)
    return codes, X


@pytest.mark.parametrize("m,n,bits", [(5, 7, 3), (8, 8, 2), (9, 4, 4), (1, 6, 3), (6, 1, 3)])
def test_quadrant_order_agrees(m, n, bits):
    """Thm. 3.1: any order that respects the dependencies gives the same
    codes and pre-rounding values as every tier."""
    W, f, g = _problem(m, n, 900 + 7 * m + n, bits=bits)
    codes, X = _quadrant_order(W, f.LA, f.LB, g)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g)
    np.testing.assert_array_equal(codes, ref.codes)
    np.testing.assert_allclose(X, ref.X, atol=1e-10)
    np.testing.assert_array_equal(O.bakron(W, f.LA, f.LB, g).codes, codes)


# --------------------------------------------------------- planted mistakes
def _alg5_original_w(W, LA, LB, grid):
    """Alg. 5 with "V - W" read as values minus the ORIGINAL input (wrong)."""
    W0 = np.asarray(W, np.float64)
    Wk = W0.copy()
    S, Z = grid.expand(W0.shape[1])
    m, n = W0.shape
    K = np.add.outer(np.arange(m), np.arange(n))
    V = np.zeros_like(W0)
    codes = np.zeros_like(W0)

    def rec(k, l):
        if l == k + 1:
            on = K == k
            c, v = O.quantize(Wk[on], S[on], Z[on], grid.qmax)
            codes[on], V[on] = c, v
            return
        h = (k + l) // 2
        rec(k, h)
        E = np.where((K >= k) & (K < h), V - W0, 0.0)
        Wk[(K >= h) & (K < l)] += (LB @ E @ LA.T)[(K >= h) & (K < l)]
        rec(h, l)

    rec(0, m + n - 1)
    return codes.astype(np.int64)


def test_planted_mistakes_are_caught():
    """Slips planted in copies of the oracle are caught by the pins above."""
    W, f, g = _problem(8, 7, 61, bits=3)
    ref = O.bakron_vectorized(W, f.A_d, f.B_d, g).codes
    # 1) the original-W misreading of Alg. 5 changes the codes
    assert (_alg5_original_w(W, f.LA, f.LB, g) != ref).any()
    # 2) a transposed factor changes the codes
    assert (O.bakron_naive(W, f.LA.T.copy(), f.LB, g).codes != ref).any()
    assert (O.bakron_recursive(W, f.LA, f.LB.T.copy(), g).codes != ref).any()
    # 2b) inside a block of the blocked tier, a transposed factor is caught too
    assert (O.bakron_recursive(W, f.LA, f.LB.T.copy(), g, base=4).codes != ref).any()
    # 3) a wrong sign on the error feedback fails the certificate
    r = O.bakron_recursive(W, -f.LA + 2 * np.eye(7), f.LB, g)
    _, bad, _ = O.certificate(W, r.codes, g, f.LA, f.LB)
    assert bad.any()


def test_row_certificate_matches_full():
    """The row-sampled certificate (RevCholesky form) equals the full one."""
    W, f, g = _problem(20, 13, 90, bits=3)
    r = O.bakron_recursive(W, f.LA, f.LB, g)
    codes = r.codes.copy()
    codes[7, 3] = (codes[7, 3] + 1) % (g.qmax + 1)        # make it fail somewhere
    Xf, badf, df = O.certificate(W, codes, g, f.LA, f.LB)
    RA, RB = O.rev_cholesky(f.A_d), O.rev_cholesky(f.B_d)
    V = O.dequantize(codes, g, 13)
    rows = np.array([0, 1, 7, 8, 19])
    D = V - W
    hi = rows.max() + 1
    Xr, badr, dr = O.certificate_rows(W[rows], codes[rows], D[:hi], O.grid_rows(g, rows), RA,
                                      RB[rows][:, :hi], rows)
    np.testing.assert_allclose(Xr, Xf[rows], atol=1e-9)
    np.testing.assert_array_equal(badr, badf[rows])
