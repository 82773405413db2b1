"""Plain float64 CPU oracle for the Kronecker factors of a Hessian.

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: nothing on the
product path imports it, and it shares no code with the CUDA library.

What it computes (Sec. 4, "Choosing the Factorization: Independence vs. Power
Iteration", and the appendix on the Hessian factorisation).  A Hessian of the
form H = E[a a^T (x) b b^T] over samples (a_t, b_t) is approximated by A (x) B:

  * K-FAC (independence):  A = E[a a^T],  B = E[b b^T];
  * Shampoo (power iteration on the rearrangement R(H) = E[vec(a a^T)
    vec(b b^T)^T], whose best rank-1 term is the best Kronecker term):
        A^(i+1) = E[tr(b^T B^(i) b) a a^T],   B^(i+1) = E[tr(a^T A^(i) a) b b^T],
    from A^(0) = I, B^(0) = I; one iteration gives the weighted Grams
        A = E[|b|^2 a a^T],  B = E[|a|^2 b b^T].

The sample matrices hold one sample per ROW (k x d, the activations' natural
tokens x features layout); a matrix-valued sample (d x r) enters as its r
columns, each a row here, all with the sample's weight.  The expectation is
the mean over the k samples.

The device primitive is the weighted Gram
    G <- beta G + alpha sum_t w_t x_t x_t^T = beta G + alpha X^T diag(w) X,
which ``gram`` writes out as that definition.
"""
from __future__ import annotations

import numpy as np

F64 = np.float64


def gram(X, w=None, alpha: float = 1.0, beta: float = 0.0, G0=None) -> np.ndarray:
    """beta G0 + alpha X^T diag(w) X in float64 (w = None: all ones)."""
    X = np.asarray(X, dtype=F64)
    k, d = X.shape
    wx = X if w is None else X * np.asarray(w, dtype=F64)[:, None]
    G = alpha * (wx.T @ X)
    if beta != 0.0:
        G = G + beta * np.asarray(G0, dtype=F64)
    return G


def sample_sqnorms(Y) -> np.ndarray:
    """|y_t|^2 per row: tr(b_t^T b_t) of a vector sample b_t = y_t."""
    Y = np.asarray(Y, dtype=F64)
    return (Y * Y).sum(axis=1)


def sample_quadforms(Y, M) -> np.ndarray:
    """y_t^T M y_t per row: tr(b_t^T M b_t) for a vector sample."""
    Y = np.asarray(Y, dtype=F64)
    return ((Y @ np.asarray(M, dtype=F64)) * Y).sum(axis=1)


def kfac_factors(a, b):
    """K-FAC: A = E[a a^T], B = E[b b^T] over k paired vector samples."""
    k = np.asarray(a).shape[0]
    return gram(a, alpha=1.0 / k), gram(b, alpha=1.0 / k)


def shampoo_factors(a, b, iterations: int = 1):
    """Shampoo: `iterations` unnormalised power-iteration steps from identity
    (Appendix, Hessian factorisation); both factors of step i + 1 use the
    factors of step i."""
    a = np.asarray(a, dtype=F64)
    b = np.asarray(b, dtype=F64)
    k = a.shape[0]
    A = np.eye(a.shape[1])
    B = np.eye(b.shape[1])
    for _ in range(iterations):
        wa = sample_quadforms(b, B)          # tr(b^T B b) weighs a a^T
        wb = sample_quadforms(a, A)          # tr(a^T A a) weighs b b^T
        A, B = gram(a, wa, alpha=1.0 / k), gram(b, wb, alpha=1.0 / k)
    return A, B


def rearranged_hessian(a, b) -> np.ndarray:
    """R(H) = E[vec(a a^T) vec(b b^T)^T] (column-major vec), formed
    explicitly; for tiny pins only."""
    a = np.asarray(a, dtype=F64)
    b = np.asarray(b, dtype=F64)
    k = a.shape[0]
    R = np.zeros((a.shape[1] ** 2, b.shape[1] ** 2))
    for t in range(k):
        R += np.outer(np.outer(a[t], a[t]).reshape(-1, order="F"),
                      np.outer(b[t], b[t]).reshape(-1, order="F"))
    return R / k


def kronecker_hessian(a, b) -> np.ndarray:
    """H = E[a a^T (x) b b^T] formed explicitly (for tiny pins only)."""
    a = np.asarray(a, dtype=F64)
    b = np.asarray(b, dtype=F64)
    return sum(np.kron(np.outer(a[t], a[t]), np.outer(b[t], b[t]))
               for t in range(a.shape[0])) / a.shape[0]
