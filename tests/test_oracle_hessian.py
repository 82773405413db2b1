"""Pins of the oracle's Kronecker-factor accumulation (Sec. 4, "Choosing the
Factorization"; appendix on the Hessian factorisation).

Each check compares the oracle with something other than itself: a
hand-computed Gram, the sum of outer products written as loops, the
explicitly formed H = E[a a^T (x) b b^T] and its rearrangement R(H), and the
SVD of R(H) that the power iteration must converge to.
"""
import numpy as np
import pytest

import oracle as O


def _loops_gram(X, w, alpha, beta, G0):
    k, d = len(X), len(X[0])
    G = [[beta * G0[i][j] for j in range(d)] for i in range(d)]
    for t in range(k):
        for i in range(d):
            for j in range(d):
                G[i][j] += alpha * w[t] * X[t][i] * X[t][j]
    return np.array(G)


def test_hand_worked_gram():
    X = np.array([[1.0, 2.0], [3.0, 4.0]])
    np.testing.assert_array_equal(O.gram(X), [[10.0, 14.0], [14.0, 20.0]])
    np.testing.assert_array_equal(O.gram(X, w=[2.0, 0.5]), [[6.5, 10.0], [10.0, 16.0]])
    G0 = np.array([[1.0, -1.0], [-1.0, 3.0]])
    np.testing.assert_array_equal(O.gram(X, alpha=0.5, beta=2.0, G0=G0),
                                  [[7.0, 5.0], [5.0, 16.0]])


def test_gram_equals_outer_product_loops():
    rng = np.random.default_rng(1)
    X = rng.normal(size=(9, 5))
    w = rng.uniform(0.1, 2.0, size=9)
    G0 = rng.normal(size=(5, 5))
    ref = _loops_gram(X.tolist(), w.tolist(), 0.3, -0.7, G0.tolist())
    np.testing.assert_allclose(O.gram(X, w, 0.3, -0.7, G0), ref, rtol=1e-13, atol=1e-13)


def test_one_hot_rows_count_weights():
    """One-hot samples: a diagonal Gram holding each feature's summed weight."""
    idx = np.array([0, 2, 2, 1, 2, 0])
    X = np.eye(3)[idx]
    w = np.array([1.0, 2.0, 3.0, 4.0, 5.0, 6.0])
    np.testing.assert_array_equal(O.gram(X, w), np.diag([7.0, 4.0, 10.0]))


def test_gram_symmetric_psd():
    rng = np.random.default_rng(2)
    X = rng.standard_t(3, size=(50, 12))
    G = O.gram(X, rng.uniform(0, 1, 50), alpha=1 / 50)
    np.testing.assert_allclose(G, G.T, rtol=1e-13, atol=1e-15)
    assert np.linalg.eigvalsh(G).min() > -1e-12


def test_sqnorms_and_quadforms():
    Y = np.array([[3.0, 4.0], [1.0, -1.0]])
    np.testing.assert_array_equal(O.sample_sqnorms(Y), [25.0, 2.0])
    M = np.array([[2.0, 1.0], [1.0, 0.0]])
    # y^T M y = 2 y0^2 + 2 y0 y1
    np.testing.assert_array_equal(O.sample_quadforms(Y, M), [42.0, 0.0])
    np.testing.assert_array_equal(O.sample_quadforms(Y, np.eye(2)), O.sample_sqnorms(Y))


def test_rearrangement_maps_kronecker_entries():
    """R(H)[j1 + n j2, i1 + m i2] = H[j1 m + i1, j2 m + i2] (column-major vec,
    a on the input side: n features, b on the output side: m)."""
    rng = np.random.default_rng(3)
    a, b = rng.normal(size=(4, 3)), rng.normal(size=(4, 2))
    n, m = 3, 2
    H = O.kronecker_hessian(a, b)
    R = O.rearranged_hessian(a, b)
    for j1 in range(n):
        for j2 in range(n):
            for i1 in range(m):
                for i2 in range(m):
                    assert R[j1 + n * j2, i1 + m * i2] == pytest.approx(
                        H[j1 * m + i1, j2 * m + i2], rel=1e-14, abs=1e-14)


def test_one_shampoo_step_is_one_power_step():
    """vec(A^(1)) = R(H) vec(I_m), vec(B^(1)) = R(H)^T vec(I_n)."""
    rng = np.random.default_rng(4)
    a, b = rng.normal(size=(7, 3)), rng.normal(size=(7, 4))
    A, B = O.shampoo_factors(a, b, 1)
    R = O.rearranged_hessian(a, b)
    np.testing.assert_allclose(A.reshape(-1, order="F"), R @ np.eye(4).reshape(-1, order="F"),
                               rtol=1e-12)
    np.testing.assert_allclose(B.reshape(-1, order="F"), R.T @ np.eye(3).reshape(-1, order="F"),
                               rtol=1e-12)
    # the weighted Grams with |b|^2 and |a|^2
    np.testing.assert_allclose(A, O.gram(a, O.sample_sqnorms(b), alpha=1 / 7), rtol=1e-13)
    np.testing.assert_allclose(B, O.gram(b, O.sample_sqnorms(a), alpha=1 / 7), rtol=1e-13)


def test_power_iteration_reaches_best_kronecker_term():
    """Many steps: vec(A), vec(B) align with the top singular pair of R(H)."""
    rng = np.random.default_rng(5)
    a, b = rng.normal(size=(20, 3)), rng.normal(size=(20, 3))
    R = O.rearranged_hessian(a, b)
    U, S, Vt = np.linalg.svd(R)
    A, B = O.shampoo_factors(a, b, 40)
    va, vb = A.reshape(-1, order="F"), B.reshape(-1, order="F")
    assert abs(va @ U[:, 0]) / np.linalg.norm(va) > 1 - 1e-10
    assert abs(vb @ Vt[0]) / np.linalg.norm(vb) > 1 - 1e-10


def test_kfac_equals_shampoo_for_constant_norms():
    """|b_t| = c for all t: the one-step Shampoo A is c^2 times K-FAC's."""
    rng = np.random.default_rng(6)
    a = rng.normal(size=(30, 4))
    b = rng.normal(size=(30, 5))
    b = 1.5 * b / np.linalg.norm(b, axis=1, keepdims=True)
    Ak, _ = O.kfac_factors(a, b)
    As, _ = O.shampoo_factors(a, b, 1)
    np.testing.assert_allclose(As, 2.25 * Ak, rtol=1e-12)


def test_planted_mistakes_are_caught():
    X = np.array([[1.0, 2.0], [3.0, 4.0]])
    w = np.array([2.0, 0.5])
    good = O.gram(X, w)
    assert not np.array_equal(X @ X.T, good)                        # X X^T instead of X^T X
    assert not np.array_equal((X * w[:, None]).T @ (X * w[:, None]), good)   # w applied twice
    assert not np.array_equal((X.T * w[:, None]) @ X, good)         # w on the wrong index
