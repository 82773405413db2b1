"""Plain, slow, float64 CPU oracle for BaKron's two-sided adaptive rounding.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code with the CUDA library and imports nothing from it.

What it computes (BaKron, Sec. 3 of the paper).  Given W (m x n) and SPD
Kronecker factors A (n x n, input side) and B (m x m, output side), run Babai
nearest-plane / GPTQ error feedback on vec(W) under the Hessian H = A (x) B
(Alg. 2 is Alg. 1 applied to vec(W); Prop. 3.1 maps it back to matrices).
The result is defined order-free by Eq. (canonical-antidiagonal) of the
equivalence proof (Appendix "Equivalence Proofs"):

    X_k = Pi_{I_k}( W + L^B (sum_{l<k} E_l) L^A^T ),  V_k = Q(X_k),  E_k = V_k - X_k

where L^A, L^B are Cholesky(A^-1), Cholesky(B^-1) with columns scaled to a
unit diagonal, and Q maps a scalar to the nearest element of the quantisation
alphabet (Sec. 3.1: "replace round by a quantize function").

Tiers (all fp64, all give the same codes by Thm. 3.1):
  * ``bakron_vectorized``   -- the definition: explicit mn x mn A (x) B,
                               Cholesky of its inverse, Alg. 1 in vec order.
  * ``bakron_naive``        -- Alg. 2 (row-major, rank-1 updates).
  * ``bakron_antidiagonal`` -- Alg. 3 (one batched update per anti-diagonal).
  * ``bakron_recursive``    -- Alg. 4 (split the longer side, bulk update);
                               with ``base`` > 1 it stops at blocks of at most
                               base x base and rounds each by Alg. 3 restricted
                               to the block (the full-size comparisons).
  * ``bakron``              -- Alg. 5 (halve the anti-diagonal range).
Plus the textbook GPTQ loop (``gptq_rows``), round-to-nearest, the
fixed-point certificate derived from the canonical definition, the objective
and the error bound of Cor. 3.3.

Readings taken where the paper is silent:
  * indices are 0-based here; the paper's are 1-based with exclusive upper
    ends (Sec. 3.1), so anti-diagonal k of the paper is i + j = k - 2 here;
  * halves use floor(n/2) for the first part (complexity proof of Alg. 4);
  * the workspace keeps pre-rounding values of processed entries and
    "V - W" in Alg. 4/5 means values minus those (equivalence proof,
    conventions paragraph);
  * factors are prepared once at top level (same paragraph);
  * the alphabet is GPTQ's asymmetric min-max grid over 2^b codes, computed
    once from the original W per row or per (row, column group), in fp32
    arithmetic so that both sides hold bit-identical scales and zeros; codes
    are c = clamp(rint(x / s) + z, 0, 2^b - 1) with round-half-to-even, the
    tie rule the proof leaves open; value v = s (c - z);
  * ``integer_grid`` is the paper's plain round() onto Z (s = 1, no clamp).
"""
from __future__ import annotations

import dataclasses
import itertools

import numpy as np
import scipy.linalg as sla

F64 = np.float64
F32 = np.float32


# ----------------------------------------------------------------------------
# Sec. 4 and Appendix "Experiments": damping of the Gram matrices.
# ----------------------------------------------------------------------------
def damped(H: np.ndarray, damp: float) -> np.ndarray:
    """H + damp * mean(diag H) * I (the paper regularises each Gram this way,
    with damp = 0.5 in its experiments; the configs here use 0.01)."""
    H = np.asarray(H, dtype=F64)
    return H + damp * np.mean(np.diag(H)) * np.eye(H.shape[0], dtype=F64)


# ----------------------------------------------------------------------------
# Sec. 3.1 notation and Alg. 1/2: factor preparation.
# ----------------------------------------------------------------------------
def unit_lower_factor(H: np.ndarray) -> np.ndarray:
    """Cholesky(H^-1), then each column divided by its diagonal entry (Alg. 1,
    first two lines).  Lower triangular with unit diagonal."""
    L = np.linalg.cholesky(np.linalg.inv(np.asarray(H, dtype=F64)))
    return L / np.diag(L)[None, :]


def rev_cholesky(H: np.ndarray) -> np.ndarray:
    """RevCholesky(H) (Sec. 3.1): the lower triangular R with R^T R = H and a
    positive diagonal.  Obtained from the ordinary Cholesky of the matrix with
    rows and columns reversed: J H J = C C^T  =>  H = (J C J)(J C J)^T, whose
    transpose pair gives R = J C^T J."""
    H = np.asarray(H, dtype=F64)
    C = np.linalg.cholesky(H[::-1, ::-1])
    return np.ascontiguousarray(C.T[::-1, ::-1])


def unit_lower_factor_via_rev(H: np.ndarray) -> np.ndarray:
    """Same matrix as ``unit_lower_factor`` without forming H^-1.

    With R = RevCholesky(H): H^-1 = R^-1 R^-T and R^-1 is lower triangular with
    a positive diagonal, so Cholesky(H^-1) = R^-1 and its unit-diagonal form is
    R^-1 diag(R).  Used for large factors; tests pin it to the definition."""
    R = rev_cholesky(H)
    Rinv = sla.solve_triangular(R, np.eye(R.shape[0]), lower=True)
    return Rinv * np.diag(R)[None, :]


@dataclasses.dataclass
class Factors:
    LA: np.ndarray   # n x n unit lower, input side
    LB: np.ndarray   # m x m unit lower, output side
    rA: np.ndarray   # diag(RevCholesky(A_d)), length n
    rB: np.ndarray   # diag(RevCholesky(B_d)), length m
    A_d: np.ndarray
    B_d: np.ndarray


def prepare(A: np.ndarray, B: np.ndarray, damp: float,
            via_inverse: bool = True) -> Factors:
    """Damp both Grams and build their unit-lower factors (done once, at the
    top level: equivalence proof, conventions paragraph)."""
    A_d, B_d = damped(A, damp), damped(B, damp)
    f = unit_lower_factor if via_inverse else unit_lower_factor_via_rev
    return Factors(f(A_d), f(B_d), np.diag(rev_cholesky(A_d)).copy(),
                   np.diag(rev_cholesky(B_d)).copy(), A_d, B_d)


# ----------------------------------------------------------------------------
# Sec. 3.1: the base quantiser that replaces round().
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class Grid:
    """Per-row (group == 0) or per-(row, group) affine grid over 2^bits codes.

    s, z have shape (m, G).  qmax is None for the unbounded integer lattice."""
    s: np.ndarray
    z: np.ndarray
    qmax: int | None
    group: int

    def expand(self, n: int):
        """Per-entry scale and zero arrays of shape (m, n)."""
        g = n if self.group == 0 else self.group
        return (np.repeat(self.s.astype(F64), g, axis=1)[:, :n],
                np.repeat(self.z.astype(F64), g, axis=1)[:, :n])


def quant_grid(W: np.ndarray, bits: int, group: int = 0) -> Grid:
    """GPTQ-style asymmetric min-max grid from the ORIGINAL W, in fp32.

    xmin = min(0, min w), xmax = max(0, max w); an all-zero row/group uses
    [-1, 1]; s = (xmax - xmin) / (2^b - 1); z = rint(-xmin / s)."""
    W = np.asarray(W, dtype=F32)
    m, n = W.shape
    g = n if group == 0 else group
    if n % g:
        raise ValueError("group must divide n")
    Wg = W.reshape(m, n // g, g)
    xmin = np.minimum(Wg.min(axis=2), F32(0))
    xmax = np.maximum(Wg.max(axis=2), F32(0))
    zero = (xmin == 0) & (xmax == 0)
    xmin = np.where(zero, F32(-1), xmin).astype(F32)
    xmax = np.where(zero, F32(1), xmax).astype(F32)
    qmax = (1 << bits) - 1
    s = ((xmax - xmin) / F32(qmax)).astype(F32)
    z = np.rint((-xmin) / s).astype(F32)
    return Grid(s, z, qmax, group)


def symmetric_candidates(amax, levels: int, shrink_steps: int) -> np.ndarray:
    """Candidate scales of the symmetric alphabet (Appendix "Experiments").

    The scale starts at the row's maximal |w| divided by l and may shrink by
    up to a factor of 2: candidate k = 0..K (K = shrink_steps) is
        t_k = fl32((2K - k) / (2K l)),   s_k = fl32(amax * t_k)
    (K = 0: the single candidate t_0 = fl32(1 / l)).  Each is one correctly
    rounded fp32 operation on exact operands, so these are bit-identical to an
    fp32 implementation.  An all-zero row/group uses amax = 1."""
    amax = F32(amax)
    if amax == 0:
        amax = F32(1)
    if shrink_steps == 0:
        t = np.array([F32(F64(1) / F64(levels))], dtype=F32)
    else:
        k = np.arange(shrink_steps + 1, dtype=F64)
        t = ((2 * shrink_steps - k) / F64(2 * shrink_steps * levels)).astype(F32)
    return (F64(amax) * t.astype(F64)).astype(F32)


def symmetric_errors(w, scales, levels: int) -> np.ndarray:
    """Squared rounding error of the values w under each candidate scale:
    sum_q (s * clamp(rint(w_q / s), -l, l) - w_q)^2, in fp64."""
    w = np.asarray(w, dtype=F32).astype(F64)
    s = np.asarray(scales, dtype=F32).astype(F64)[:, None]
    c = np.clip(np.rint(w[None, :] / s), -levels, levels)
    return ((s * c - w[None, :]) ** 2).sum(axis=1)


def symmetric_grid(W: np.ndarray, levels: int, group: int = 0,
                   shrink_steps: int = 50) -> Grid:
    """The paper's experimental alphabet (Appendix "Experiments"): codes
    {-l, ..., +l} per row (or per (row, group)), scale = max |w| / l shrunk by
    the candidate factor in [1/2, 1] (``symmetric_candidates``) whose
    round-to-nearest squared error over the row is least (the first such
    candidate, i.e. the largest scale, on exact ties).  Expressed in the
    affine form of ``Grid``: z = l, qmax = 2 l, so code c stands for the
    integer c - l and value s (c - l)."""
    W = np.asarray(W, dtype=F32)
    m, n = W.shape
    g = n if group == 0 else group
    if n % g:
        raise ValueError("group must divide n")
    G = n // g
    s = np.empty((m, G), dtype=F32)
    for i in range(m):
        for j in range(G):
            w = W[i, j * g:(j + 1) * g]
            cand = symmetric_candidates(np.abs(w).max(), levels, shrink_steps)
            err = symmetric_errors(w, cand, levels)
            s[i, j] = cand[int(np.argmin(err))]
    return Grid(s, np.full((m, G), F32(levels)), 2 * levels, group)


def integer_grid(m: int) -> Grid:
    """The paper's plain round() onto Z: s = 1, z = 0, no clamping."""
    return Grid(np.ones((m, 1), F32), np.zeros((m, 1), F32), None, 0)


def quantize(x, s, z, qmax):
    """Nearest alphabet element: code c = clamp(rint(x/s) + z, 0, qmax) with
    round-half-to-even, value v = s (c - z).  Works on scalars and arrays."""
    c = np.rint(np.asarray(x, dtype=F64) / s) + z
    if qmax is not None:
        c = np.clip(c, 0, qmax)
    return c, s * (c - z)


def midpoint_distance(x, s):
    """Distance, in grid units, from x/s to the nearest half-integer, i.e. to
    the nearest rounding boundary."""
    t = np.asarray(x, dtype=F64) / s
    return np.abs(t - np.floor(t) - 0.5)


@dataclasses.dataclass
class Result:
    codes: np.ndarray   # int64 (m, n)
    V: np.ndarray       # quantised values s (c - z)
    X: np.ndarray       # pre-rounding values (the workspace after the solve)

    @property
    def E(self):
        return self.V - self.X


def _setup(W, grid):
    W = np.asarray(W, dtype=F64)
    S, Z = grid.expand(W.shape[1])
    return W.copy(), S, Z


# ----------------------------------------------------------------------------
# Alg. 1 (GPTQ on one vector) applied to vec(W) with H = A (x) B: the definition.
# ----------------------------------------------------------------------------
def bakron_vectorized(W, A_d, B_d, grid: Grid) -> Result:
    """Alg. 2's meaning written out literally: vec(W) column-major (Sec. 3.1),
    H = A_d (x) B_d formed explicitly (mn x mn), L = Cholesky(H^-1) with unit
    columns, then Alg. 1's sequential loop.  Only for tiny m*n."""
    W, S, Z = _setup(W, grid)
    m, n = W.shape
    H = np.kron(np.asarray(A_d, F64), np.asarray(B_d, F64))
    L = unit_lower_factor(H)
    w = W.reshape(-1, order="F").copy()
    s = S.reshape(-1, order="F")
    z = Z.reshape(-1, order="F")
    x_pre = np.zeros_like(w)
    codes = np.zeros_like(w)
    for i in range(m * n):
        x_pre[i] = w[i]
        c, v = quantize(w[i], s[i], z[i], grid.qmax)
        codes[i] = c
        w[i:] += (v - w[i]) * L[i:, i]          # w <- w + Delta * L_i
    shape = (m, n)
    return Result(codes.reshape(shape, order="F").astype(np.int64),
                  w.reshape(shape, order="F"),
                  x_pre.reshape(shape, order="F"))


# ----------------------------------------------------------------------------
# Alg. 2: BaKron-naive.
# ----------------------------------------------------------------------------
def bakron_naive(W, LA, LB, grid: Grid) -> Result:
    """Row-major double loop with the rank-1 update W += L^B_i Delta L^A_j^T.
    The update is applied to the block W[i:, j:] only, which is where the
    lower-triangular columns L^B_i, L^A_j are nonzero."""
    W, S, Z = _setup(W, grid)
    m, n = W.shape
    X = np.zeros_like(W)
    codes = np.zeros_like(W)
    for i in range(m):
        for j in range(n):
            X[i, j] = W[i, j]
            c, v = quantize(W[i, j], S[i, j], Z[i, j], grid.qmax)
            codes[i, j] = c
            W[i:, j:] += (v - W[i, j]) * np.outer(LB[i:, i], LA[j:, j])
    return Result(codes.astype(np.int64), W, X)


# ----------------------------------------------------------------------------
# Alg. 3: BaKron-antidiagonal.
# ----------------------------------------------------------------------------
def bakron_antidiagonal(W, LA, LB, grid: Grid) -> Result:
    """For each anti-diagonal: round it whole, then W += L^B Delta L^A^T."""
    W, S, Z = _setup(W, grid)
    m, n = W.shape
    K = np.add.outer(np.arange(m), np.arange(n))
    X = np.zeros_like(W)
    codes = np.zeros_like(W)
    for k in range(m + n - 1):
        on = K == k
        X[on] = W[on]
        c, v = quantize(W[on], S[on], Z[on], grid.qmax)
        codes[on] = c
        delta = np.zeros_like(W)
        delta[on] = v - W[on]
        W += LB @ delta @ LA.T
    return Result(codes.astype(np.int64), W, X)


# ----------------------------------------------------------------------------
# Alg. 4: BaKron-recursive (divide and conquer on the longer side).
# ----------------------------------------------------------------------------
def bakron_recursive(W, LA, LB, grid: Grid, base: int = 1) -> Result:
    """Split columns if m < n else rows (first part floor(size/2)); solve the
    first part; W_2 += L^B (V_1 - W_1) L^A_21^T (column split) or
    L^B_21 (V_1 - W_1) L^A^T (row split); solve the second part.  The
    workspace W is shared in place and keeps pre-rounding values.

    ``base`` (default 1: Alg. 4 down to single entries) stops the splitting at
    blocks with at most ``base`` rows and ``base`` columns and rounds such a
    block by Alg. 3 restricted to it: for each of its anti-diagonals, round the
    entries, then add L^B_blk Delta L^A_blk^T to the block's later entries
    (Delta: the errors of that anti-diagonal).  Inside a block only entries
    up-left of an entry feed it, so this is the same problem Alg. 4 would solve
    there, and by Thm. 3.1 every order gives the same codes; it only trades
    the recursion's many tiny calls for a few anti-diagonal steps, which keeps
    full-size problems within minutes."""
    Wk, S, Z = _setup(W, grid)
    m, n = Wk.shape
    V = np.zeros_like(Wk)
    codes = np.zeros_like(Wk)
    qmax = grid.qmax

    diagonals = {}

    def antidiagonals(mm, nn):
        """Row and column indices of each anti-diagonal of an mm x nn block."""
        if (mm, nn) not in diagonals:
            i, j = np.divmod(np.arange(mm * nn), nn)
            order = np.argsort(i + j, kind="stable")
            k = (i + j)[order]
            cuts = np.searchsorted(k, np.arange(mm + nn))
            diagonals[(mm, nn)] = [(i[order][a:b], j[order][a:b])
                                   for a, b in zip(cuts[:-1], cuts[1:])]
        return diagonals[(mm, nn)]

    def block(r0, r1, c0, c1):
        LBb, LAb = LB[r0:r1, r0:r1], LA[c0:c1, c0:c1]
        Wb, Sb, Zb = Wk[r0:r1, c0:c1], S[r0:r1, c0:c1], Z[r0:r1, c0:c1]
        Cb, Vb = codes[r0:r1, c0:c1], V[r0:r1, c0:c1]
        for ii, jj in antidiagonals(r1 - r0, c1 - c0):
            x = Wb[ii, jj]
            c, v = quantize(x, Sb[ii, jj], Zb[ii, jj], qmax)
            Cb[ii, jj] = c
            Vb[ii, jj] = v
            # W_blk += L^B_blk Delta L^A_blk^T with Delta = v - x on this
            # anti-diagonal: the sum of its columns' outer products.  Earlier
            # entries receive exact zeros (the factors are lower triangular);
            # the rounded entries themselves keep their pre-rounding values.
            Wb += (LBb[:, ii] * (v - x)) @ LAb[:, jj].T
            Wb[ii, jj] = x

    def rec(r0, r1, c0, c1):
        mm, nn = r1 - r0, c1 - c0
        if mm == 1 and nn == 1:
            c, v = quantize(Wk[r0, c0], S[r0, c0], Z[r0, c0], qmax)
            codes[r0, c0] = c
            V[r0, c0] = v
            return
        if base > 1 and mm <= base and nn <= base:
            block(r0, r1, c0, c1)
            return
        if mm < nn:
            h = c0 + nn // 2
            rec(r0, r1, c0, h)
            E = V[r0:r1, c0:h] - Wk[r0:r1, c0:h]
            Wk[r0:r1, h:c1] += LB[r0:r1, r0:r1] @ E @ LA[h:c1, c0:h].T
            rec(r0, r1, h, c1)
        else:
            h = r0 + mm // 2
            rec(r0, h, c0, c1)
            E = V[r0:h, c0:c1] - Wk[r0:h, c0:c1]
            Wk[h:r1, c0:c1] += LB[h:r1, r0:h] @ E @ LA[c0:c1, c0:c1].T
            rec(h, r1, c0, c1)

    rec(0, m, 0, n)
    return Result(codes.astype(np.int64), V, Wk)


# ----------------------------------------------------------------------------
# Alg. 5: BaKron (recursive halving of the anti-diagonal range).
# ----------------------------------------------------------------------------
def bakron(W, LA, LB, grid: Grid) -> Result:
    """rec(k, l): a single anti-diagonal is rounded at its workspace values;
    otherwise h = floor((k + l)/2), rec(k, h), then
    W += antidiag_{h:l}( L^B (V - antidiag_{k:h}(W)) L^A^T ), then rec(h, l)."""
    Wk, S, Z = _setup(W, grid)
    m, n = Wk.shape
    K = np.add.outer(np.arange(m), np.arange(n))
    V = np.zeros_like(Wk)
    codes = np.zeros_like(Wk)

    def rec(k, l):
        if l == k + 1:
            on = K == k
            c, v = quantize(Wk[on], S[on], Z[on], grid.qmax)
            codes[on] = c
            V[on] = v
            return
        h = (k + l) // 2
        rec(k, h)
        first = (K >= k) & (K < h)
        second = (K >= h) & (K < l)
        E = np.where(first, V - Wk, 0.0)
        U = LB @ E @ LA.T
        Wk[second] += U[second]
        rec(h, l)

    rec(0, m + n - 1)
    return Result(codes.astype(np.int64), V, Wk)


# ----------------------------------------------------------------------------
# Textbook GPTQ (Frantar et al.), for the B = I special case (Sec. 1, Sec. 3.6).
# ----------------------------------------------------------------------------
def gptq_rows(W, H, S, Z, qmax) -> Result:
    """GPTQ as its own paper states it, per row of W under Hessian H, with
    per-entry scale S and zero Z (arrays shaped like W): U = upper Cholesky
    factor of H^-1; for column i: quantise, divide the error by U_ii and
    subtract err * U[i, i:] from the remaining columns."""
    Wk = np.asarray(W, dtype=F64).copy()
    S = np.asarray(S, F64)
    Z = np.asarray(Z, F64)
    m, n = Wk.shape
    U = np.linalg.cholesky(np.linalg.inv(np.asarray(H, F64))).T
    codes = np.zeros_like(Wk)
    Q = np.zeros_like(Wk)
    X = np.zeros_like(Wk)
    for i in range(n):
        X[:, i] = Wk[:, i]
        c, q = quantize(Wk[:, i], S[:, i], Z[:, i], qmax)
        codes[:, i] = c
        Q[:, i] = q
        err = (Wk[:, i] - q) / U[i, i]
        Wk[:, i:] -= np.outer(err, U[i, i:])
    return Result(codes.astype(np.int64), Q, X)


def rtn(W, grid: Grid) -> Result:
    """Round-to-nearest onto the same grid (no error feedback)."""
    Wk, S, Z = _setup(W, grid)
    c, v = quantize(Wk, S, Z, grid.qmax)
    return Result(c.astype(np.int64), v, Wk)


def dequantize(codes, grid: Grid, n: int) -> np.ndarray:
    S, Z = grid.expand(n)
    return S * (np.asarray(codes, F64) - Z)


# ----------------------------------------------------------------------------
# Fixed-point certificate, objective and error bound.
# ----------------------------------------------------------------------------
def teacher_forced(W, V, LA, LB):
    """Pre-rounding values implied by a candidate V.

    From the canonical definition, V = W + L^B E L^A^T with E the committed
    errors (an entry's own term enters with the unit diagonal, all others with
    i + j smaller).  Hence E = L^B^-1 (V - W) L^A^-T and X = V - E: X[p, q] is
    the value entry (p, q) is rounded at given the decisions V makes on every
    entry before it.  V is BaKron's output iff V = Q(X) entrywise."""
    D = np.asarray(V, F64) - np.asarray(W, F64)
    Y = sla.solve_triangular(LB, D, lower=True, unit_diagonal=True)
    E = sla.solve_triangular(LA, Y.T, lower=True, unit_diagonal=True).T
    return np.asarray(V, F64) - E, E


def certificate(W, codes, grid: Grid, LA, LB):
    """Check codes against the canonical definition, entry by entry.

    Returns (X, mismatch mask, midpoint distance of X in grid units)."""
    W = np.asarray(W, F64)
    n = W.shape[1]
    S, Z = grid.expand(n)
    V = S * (np.asarray(codes, F64) - Z)
    X, _ = teacher_forced(W, V, LA, LB)
    c, _ = quantize(X, S, Z, grid.qmax)
    return X, c != codes, midpoint_distance(X, S)


def objective(W, V, A_d, B_d) -> float:
    """tr((W - V)^T B (W - V) A) = vec(W - V)^T (A (x) B) vec(W - V)."""
    D = np.asarray(W, F64) - np.asarray(V, F64)
    return float(np.sum((B_d @ D) * (D @ A_d)))


def objective_from_errors(E, rA, rB) -> float:
    """The same objective from the committed errors: with R = RevCholesky,
    R (V - W) R'^T = diag(rB) E diag(rA) (because L^-1 = diag(R)^-1 R)."""
    return float(np.sum((np.asarray(rB)[:, None] * E * np.asarray(rA)[None, :]) ** 2))


def error_bound(grid: Grid, rA, rB, n: int) -> float:
    """Cor. 3.3 with per-entry step s: 1/4 sum_pq s_pq^2 rB_p^2 rA_q^2
    (valid while no entry is clamped)."""
    S, _ = grid.expand(n)
    return 0.25 * float(np.sum((S * np.asarray(rB)[:, None] * np.asarray(rA)[None, :]) ** 2))


# ----------------------------------------------------------------------------
# Brute force on tiny inputs.
# ----------------------------------------------------------------------------
def brute_force(W, LA, LB, A_d, B_d, grid: Grid):
    """Enumerate every code matrix over the finite alphabet.

    Returns (list of fixed points of the certificate, minimal objective)."""
    W = np.asarray(W, F64)
    m, n = W.shape
    if grid.qmax is None:
        raise ValueError("brute force needs a finite alphabet")
    fixed = []
    best = np.inf
    for flat in itertools.product(range(grid.qmax + 1), repeat=m * n):
        codes = np.array(flat, dtype=np.int64).reshape(m, n)
        V = dequantize(codes, grid, n)
        best = min(best, objective(W, V, A_d, B_d))
        _, bad, _ = certificate(W, codes, grid, LA, LB)
        if not bad.any():
            fixed.append(codes)
    return fixed, best


def babai_step_by_enumeration(x, s, z, qmax):
    """Per-coordinate Babai step as an argmin over the alphabet (ties to the
    even code, matching round-half-to-even)."""
    cands = np.arange(qmax + 1, dtype=F64)
    d = np.abs(s * (cands - z) - x)
    best = d.min()
    idx = np.flatnonzero(np.isclose(d, best, rtol=0, atol=1e-15 * max(1.0, abs(x))))
    if len(idx) > 1:
        even = [i for i in idx if (int(cands[i] - z) % 2) == 0]
        return int(cands[even[0]] if even else cands[idx[0]])
    return int(cands[idx[0]])


def certificate_rows(W_rows, codes_rows, D_rows_above, grid_rows, RA, RB_rows, rows):
    """The certificate on a subset of rows, from RevCholesky factors.

    With L^-1 = diag(R)^-1 R (R = RevCholesky), E = diag(R_B)^-1 R_B (V - W)
    R_A^T diag(R_A)^-1.  For a set of rows P, (R_B (V - W))[P] needs R_B[P, :]
    and (V - W) on rows 0..max(P) only, so large problems are checked on
    sampled row blocks without the full m x m solve.
      W_rows, codes_rows : W and codes on rows P (|P| x n)
      D_rows_above       : (V - W) on rows 0..max(P) (as needed by R_B[P, :])
      grid_rows          : Grid restricted to rows P
      RA                 : RevCholesky(A_d), n x n
      RB_rows            : R_B[P, 0:max(P)+1]
      rows               : the row indices P
    Returns (X on P, mismatch mask, midpoint distance) like ``certificate``."""
    n = W_rows.shape[1]
    S, Z = grid_rows.expand(n)
    rbd = np.array([RB_rows[k, r] for k, r in enumerate(rows)], dtype=F64)
    Y = (RB_rows @ D_rows_above) / rbd[:, None]            # diag(R_B)^-1 R_B (V - W), rows P
    E = (Y @ RA.T) / np.diag(RA)[None, :]
    V = S * (np.asarray(codes_rows, F64) - Z)
    X = V - E
    c, _ = quantize(X, S, Z, grid_rows.qmax)
    return X, c != codes_rows, midpoint_distance(X, S)


def grid_rows(grid: Grid, rows) -> Grid:
    return Grid(grid.s[rows], grid.z[rows], grid.qmax, grid.group)
