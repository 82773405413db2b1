"""The B = I path (GPTQ), bakron_solve_gptq, through the C ABI.

GPTQ is BaKron with B = I (Sec. 1): every row is Alg. 1 under H = A, and the
rows are independent.  The GPU's codes are compared with the oracle's textbook
GPTQ loop (upper Cholesky of H^-1, error / U_ii, as GPTQ states Alg. 1) on the
same rows under H = (L L^T)^-1, whose updates are exactly the unit-lower factor
L the GPU was given; on ragged shapes that span several leaf launches and
tensor-core column bands, bit widths 2-8 and column groups.  At 4096 x 4096
(the attention-projection workload's W and input-side Gram) the GPU solve with
its own device prepare is compared free-running with the oracle's own fp64
solve: with B = I a near-tie decided differently can only disturb the rest of
its own row, so the parity bar (>= 99.9% identical codes, every first
difference a tie, objective within 1e-4) applies as stated.
"""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests._helpers import TIE_BAND, compare_codes, oracle_factors_fp32, root_mismatches, to_np

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    P.lib()


def _gptq_small(m, n, seed, bits, group):
    W, A, B = WL.small_problem(m, n, seed)
    f, LA32, _ = oracle_factors_fp32(A, B, 0.01)
    dev = "cuda"
    fac = P.bakron_set_factors(torch.from_numpy(LA32).to(dev), torch.eye(m, device=dev))
    codes, scales, zeros, X = P.bakron_solve_gptq(W.to(dev), fac, bits, group, prerounding=True)
    torch.cuda.synchronize()
    W64 = to_np(W)
    g = O.quant_grid(W64, bits, group)
    np.testing.assert_array_equal(scales.cpu().numpy(), g.s)
    np.testing.assert_array_equal(zeros.cpu().numpy(), g.z)
    S, Z = g.expand(n)
    LA = LA32.astype(np.float64)
    H = np.linalg.inv(LA @ LA.T)
    gp = O.gptq_rows(W64, H, S, Z, g.qmax)
    got = codes.cpu().numpy().astype(np.int64)
    st = compare_codes(W64, got, g, LA, np.eye(m), gp.codes)
    return st, got, gp, X.cpu().numpy().astype(np.float64), S, W, fac


@pytest.mark.parametrize("m,n,bits,group", [
    (1, 1, 4, 0), (33, 64, 4, 0), (70, 100, 3, 0), (96, 416, 4, 32), (130, 1000, 2, 0),
    (257, 512, 8, 64), (40, 129, 1, 0)])
def test_gptq_matches_textbook_gptq(m, n, bits, group):
    st, got, gp, X, S, _, _ = _gptq_small(m, n, 900 + m + n, bits, group)
    assert st["cert_mismatch_outside_band"] == 0, st
    if st["cert_mismatch"] == 0:
        assert st["raw_match"] == 1.0, st
        # the values each entry was rounded at, in grid units
        assert np.max(np.abs(X - gp.X) / S) < 1e-4
    else:   # a certified tie: the first differences of each row are ties
        bad = got != gp.codes
        roots = root_mismatches(bad)
        assert (O.midpoint_distance(gp.X, S)[roots] < TIE_BAND).all()


def test_gptq_equals_general_solve_with_identity_b():
    """The column schedule and the general two-sided schedule (with L^B = I)
    reach the same codes."""
    st, got, _, _, _, W, fac = _gptq_small(160, 608, 4242, 4, 0)
    general = P.bakron_solve(W.cuda(), fac, 4, 0)[0].cpu().numpy().astype(np.int64)
    assert (general == got).mean() == 1.0


def test_gptq_rejects_groups_that_split_tiles_and_reports_nonfinite():
    fac = P.bakron_set_factors(torch.eye(64, device="cuda"), torch.eye(8, device="cuda"))
    W = torch.randn(8, 64, device="cuda")
    with pytest.raises(P.BakronError) as e:
        P.bakron_solve_gptq(W, fac, 4, group_size=16)
    assert e.value.status == 1
    W[3, 7] = float("nan")
    with pytest.raises(P.BakronError) as e:
        P.bakron_solve_gptq(W, fac, 4)
    assert e.value.status == 6
    W[3, 7] = 0.0
    codes = P.bakron_solve_gptq(W, fac, 4)[0]
    assert codes.shape == (8, 64)


def test_gptq_fullsize_free_running():
    """4096 x 4096, device prepare of (A, I), against the oracle's own fp64
    solve with its own factors (Alg. 4 with the Alg. 3 base case, L^B = I)."""
    cfg = WL.CONFIGS[2]
    W, A, _ = WL.make(cfg, device="cuda")
    m, n = cfg.m, cfg.n
    I_m = torch.eye(m, device="cuda")
    ws = P.alloc_workspace(m, n)
    fac = P.bakron_prepare(A, I_m, cfg.damp, workspace=ws)
    codes = P.bakron_solve_gptq(W, fac, cfg.bits, 0, workspace=ws)[0]
    torch.cuda.synchronize()
    got = codes.cpu().numpy().astype(np.int64)
    W64, A64 = to_np(W.float()), to_np(A)
    del ws, fac, codes
    torch.cuda.empty_cache()
    f = O.prepare(A64, np.eye(m), cfg.damp, via_inverse=False)
    g = O.quant_grid(W64, cfg.bits, 0)
    ref = O.bakron_recursive(W64, f.LA, np.eye(m), g, base=64)
    bad = got != ref.codes
    roots = root_mismatches(bad)
    S, _ = g.expand(n)
    dist = O.midpoint_distance(ref.X, S)
    obj_ref = O.objective(W64, ref.V, f.A_d, f.B_d)
    obj_gpu = O.objective(W64, O.dequantize(got, g, n), f.A_d, f.B_d)
    match = 1.0 - bad.mean()
    print(f"GPTQ_FULLSIZE match={match:.6f} mismatches={int(bad.sum())} roots={int(roots.sum())} "
          f"rel_obj={abs(obj_gpu - obj_ref) / obj_ref:.3e}")
    assert (dist[roots] < TIE_BAND).all()
    assert match >= 0.999
    assert abs(obj_gpu - obj_ref) <= 1e-4 * obj_ref
