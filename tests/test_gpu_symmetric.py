"""GPU parity of the paper's experimental quantiser (Appendix "Experiments"):
the symmetric alphabet {-l..l} with an MSE-shrunk max-abs scale per row
(bakron_grid_symmetric), and the solve onto a caller's grid
(bakron_solve_with_grid), against the float64 oracle.

The scale search is an argmin over candidates whose errors the GPU sums in
fp32: its candidate scales must be the oracle's bit for bit, and its choice
must be the oracle's except where the oracle's own errors of the two choices
agree to 1e-5 relative (either is then a least-error candidate).
"""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests._helpers import TIE_BAND, compare_codes, oracle_factors_fp32, to_np

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    P.lib()


def _heavy(m, n, seed, scale=0.02):
    rng = np.random.default_rng(seed)
    return (scale * rng.standard_t(4, size=(m, n))).astype(np.float32)


def _check_grid(W32, s_gpu, z_gpu, levels, group, K):
    m, n = W32.shape
    gs = n if group == 0 else group
    assert np.all(z_gpu == levels)
    ref = O.symmetric_grid(W32, levels, group=group, shrink_steps=K)
    differ = 0
    for i in range(m):
        for j in range(n // gs):
            w = W32[i, j * gs:(j + 1) * gs]
            cand = O.symmetric_candidates(np.abs(w).max(), levels, K)
            hit = np.flatnonzero(cand == s_gpu[i, j])
            assert len(hit) == 1, (i, j, s_gpu[i, j])        # a candidate, bit for bit
            if s_gpu[i, j] != ref.s[i, j]:
                err = O.symmetric_errors(w, cand, levels)
                k_ref = int(np.flatnonzero(cand == ref.s[i, j])[0])
                assert err[hit[0]] <= err[k_ref] * (1 + 1e-5) + 1e-30, (i, j)
                differ += 1
    return differ, ref


@pytest.mark.parametrize("wdtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("levels,group,K", [(3, 0, 50), (3, 200, 50), (1, 0, 8), (7, 40, 64),
                                            (3, 0, 0)])
def test_grid_symmetric_matches_oracle(wdtype, levels, group, K):
    m, n = 37, 1000
    W = torch.from_numpy(_heavy(m, n, 17 + levels + group + K)).to("cuda", wdtype)
    W[5].zero_()                                   # all-zero row: amax = 1
    s, z = P.bakron_grid_symmetric(W, levels, group, K)
    torch.cuda.synchronize()
    W32 = W.float().cpu().numpy()
    differ, ref = _check_grid(W32, s.cpu().numpy(), z.cpu().numpy(), levels, group, K)
    assert differ <= max(1, s.numel() // 100)
    if K == 0:
        np.testing.assert_array_equal(s.cpu().numpy(), ref.s)
    np.testing.assert_array_equal(s.cpu().numpy()[5], ref.s[5])


def test_grid_symmetric_hand_solved_row():
    """w = (1, 1/2, 1/2, 1/2), l = 1, 8 steps: s = 5/8 (worked in the oracle's
    pins); padded to a ragged 300 columns of zeros, which add no error at any
    scale."""
    W = torch.zeros(3, 300, device="cuda")
    W[:, :4] = torch.tensor([1.0, 0.5, 0.5, 0.5], device="cuda")
    W[1] *= -1
    s, z = P.bakron_grid_symmetric(W, 1, 0, 8)
    assert s.cpu().tolist() == [[0.625], [0.625], [0.625]]
    assert z.cpu().tolist() == [[1.0], [1.0], [1.0]]


def test_grid_symmetric_strided_rows():
    W = torch.from_numpy(_heavy(20, 320, 5)).cuda()
    Wv = W[:, :300]                                # ldw 320, n 300
    s, z = P.bakron_grid_symmetric(Wv, 3, 0, 50)
    s2, _ = P.bakron_grid_symmetric(Wv.contiguous(), 3, 0, 50)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(s.cpu().numpy(), s2.cpu().numpy())


def _factors(A, B, damp):
    f, LA32, LB32 = oracle_factors_fp32(A, B, damp)
    fac = P.bakron_set_factors(torch.from_numpy(LA32).cuda(), torch.from_numpy(LB32).cuda(),
                               torch.from_numpy(f.rA.astype(np.float32)).cuda(),
                               torch.from_numpy(f.rB.astype(np.float32)).cuda())
    return f, LA32.astype(np.float64), LB32.astype(np.float64), fac


@pytest.mark.parametrize("m,n,levels,group", [(33, 65, 3, 0), (97, 131, 3, 0), (64, 96, 7, 32),
                                              (130, 256, 1, 128)])
def test_solve_with_symmetric_grid_matches_oracle(m, n, levels, group):
    W, A, B = WL.small_problem(m, n, 5000 + m + n)
    f, LA, LB, fac = _factors(A, B, 0.5)            # the paper's damping for its runs
    Wd = W.cuda()
    s, z = P.bakron_grid_symmetric(Wd, levels, group, 50)
    codes, X = P.bakron_solve_with_grid(Wd, fac, s, z, 2 * levels, group, prerounding=True)
    torch.cuda.synchronize()
    W64 = to_np(W)
    W32 = W.numpy()
    _check_grid(W32, s.cpu().numpy(), z.cpu().numpy(), levels, group, 50)
    g = O.Grid(s.cpu().numpy(), z.cpu().numpy(), 2 * levels, group)   # the GPU's (checked) grid
    ref = O.bakron_recursive(W64, LA, LB, g)
    c = codes.cpu().numpy().astype(np.int64)
    assert c.min() >= 0 and c.max() <= 2 * levels
    st = compare_codes(W64, c, g, LA, LB, ref.codes)
    assert st["cert_mismatch_outside_band"] == 0, st
    if st["cert_mismatch"] == 0:
        np.testing.assert_array_equal(c, ref.codes)
        S, _ = g.expand(n)
        assert (np.abs(X.cpu().numpy() - ref.X) / S).max() < TIE_BAND
    V = O.dequantize(c, g, n)
    o_gpu = O.objective(W64, V, f.A_d, f.B_d)
    o_ref = O.objective(W64, ref.V, f.A_d, f.B_d)
    # after a decision inside the tie band the solve follows another, equally
    # valid path: the objective then stays within 1e-3
    assert abs(o_gpu - o_ref) <= (1e-4 if st["cert_mismatch"] == 0 else 1e-3) * o_ref
    o_rtn = O.objective(W64, O.rtn(W64, g).V, f.A_d, f.B_d)
    assert o_gpu < o_rtn


@pytest.mark.parametrize("bits,group", [(4, 0), (3, 32)])
def test_solve_with_grid_reproduces_solve(bits, group):
    """The min-max grid bakron_solve computes, handed back through
    bakron_solve_with_grid, gives the same codes and pre-rounding values bit
    for bit (the same kernels in the same order)."""
    W, A, B = WL.small_problem(160, 224, 61)
    _, _, _, fac = _factors(A, B, 0.01)
    Wd = W.cuda().to(torch.bfloat16)
    codes, s, z, X = P.bakron_solve(Wd, fac, bits, group, prerounding=True)
    codes2, X2 = P.bakron_solve_with_grid(Wd, fac, s, z, (1 << bits) - 1, group,
                                          prerounding=True)
    torch.cuda.synchronize()
    assert torch.equal(codes, codes2)
    assert torch.equal(X, X2)


def test_symmetric_grid_full_size_certificate():
    """The 4096 x 4096 attention-projection weights (bf16) with l = 3 (the
    paper's setting): grid checked on 256 sampled rows, the whole solve by the
    teacher-forced certificate, and the objective below round-to-nearest on
    the same grid."""
    cfg = WL.CONFIGS[2]
    W, A, B = WL.make(cfg, device="cuda")
    ws = P.alloc_workspace(cfg.m, cfg.n)
    fac = P.bakron_prepare(A, B, cfg.damp, workspace=ws)
    s, z = P.bakron_grid_symmetric(W, 3, 0, 50)
    codes = P.bakron_solve_with_grid(W, fac, s, z, 6, 0, workspace=ws)
    torch.cuda.synchronize()
    m, n = W.shape
    sc, zc = s.cpu().numpy(), z.cpu().numpy()
    W32 = W.float().cpu().numpy()
    rows = np.random.default_rng(0).choice(m, 256, replace=False)
    _check_grid(W32[rows], sc[rows], zc[rows], 3, 0, 50)
    c = codes.cpu().numpy().astype(np.int64)
    assert c.min() >= 0 and c.max() <= 6
    g = O.Grid(sc, zc, 6, 0)
    W64 = W32.astype(np.float64)
    A_d, B_d = O.damped(to_np(A), cfg.damp), O.damped(to_np(B), cfg.damp)
    RA, RB = O.rev_cholesky(A_d), O.rev_cholesky(B_d)
    P_ = np.arange(m)
    X, bad, dist = O.certificate_rows(W64, c, O.dequantize(c, g, n) - W64, g, RA, RB, P_)
    assert int((bad & (dist >= TIE_BAND)).sum()) == 0
    assert int(bad.sum()) <= 1e-3 * bad.size
    E = O.dequantize(c, g, n) - X
    obj = O.objective_from_errors(E, np.diag(RA), np.diag(RB))
    assert obj < O.objective(W64, O.rtn(W64, g).V, A_d, B_d)
