"""Full-size parity on the five workload configs, through the C ABI, in the
launch configuration bench.py times (device prepare, then device solve).

At these sizes a free-running comparison with the fp64 oracle is not
meaningful: the error feedback is chaotic (the factors' column sums are
~10-50, so one near-tie decided differently cascades through everything to its
lower right; see the cascade measurement in the design notes).  The check is
the teacher-forced certificate, which holds at any size: the oracle computes,
in fp64 from W, A and B alone, the value every entry must be rounded at given
the codes before it (canonical definition of the equivalence proof), and
every GPU code must equal that value's rounding unless the value lies within
1e-4 grid units of a rounding boundary.  Configs 2-4 are checked on every
row; config 5 on its first 256 rows, 256 rows from the middle of B's factor
(14336..14591) and its last 64 rows.
"""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests._helpers import TIE_BAND, to_np

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    P.lib()


def _run(c):
    cfg = WL.CONFIGS[c]
    W, A, B = WL.make(cfg, device="cuda")
    ws = P.alloc_workspace(cfg.m, cfg.n)
    fac = P.bakron_prepare(A, B, cfg.damp, workspace=ws)
    codes, scales, zeros = P.bakron_solve(W, fac, cfg.bits, cfg.group, workspace=ws)
    torch.cuda.synchronize()
    out = dict(cfg=cfg, W=to_np(W.float()), A=to_np(A), B=to_np(B),
               codes=codes.cpu().numpy().astype(np.int64), scales=scales.cpu().numpy(),
               zeros=zeros.cpu().numpy())
    del ws, fac
    torch.cuda.empty_cache()
    return out


def _check(r, rows=None):
    cfg = r["cfg"]
    W64, codes = r["W"], r["codes"]
    g = O.quant_grid(W64, cfg.bits, cfg.group)
    np.testing.assert_array_equal(r["scales"], g.s)
    np.testing.assert_array_equal(r["zeros"], g.z)
    A_d, B_d = O.damped(r["A"], cfg.damp), O.damped(r["B"], cfg.damp)
    RA, RB = O.rev_cholesky(A_d), O.rev_cholesky(B_d)
    m, n = W64.shape
    blocks = [np.arange(m)] if rows is None else rows
    bad_all = tie_all = tot = 0
    obj_gpu = obj_rtn = 0.0
    for P_ in blocks:
        hi = int(P_.max()) + 1
        V_above = O.dequantize(codes[:hi], O.grid_rows(g, np.arange(hi)), n)
        D = V_above - W64[:hi]
        gr = O.grid_rows(g, P_)
        X, bad, dist = O.certificate_rows(W64[P_], codes[P_], D, gr, RA, RB[P_][:, :hi], P_)
        bad_all += int((bad & (dist >= TIE_BAND)).sum())
        tie_all += int(bad.sum())
        tot += bad.size
        if rows is None:
            E = O.dequantize(codes, g, n) - X
            obj_gpu = O.objective_from_errors(E, np.diag(RA), np.diag(RB))
            obj_rtn = O.objective(W64, O.rtn(W64, g).V, A_d, B_d)
    assert bad_all == 0, f"{bad_all} codes disagree outside the tie band"
    assert tie_all <= 1e-3 * tot
    if rows is None:
        assert obj_gpu < obj_rtn
        # objective identity at full size: trace form == error form
        V = O.dequantize(codes, g, n)
        assert O.objective(W64, V, A_d, B_d) == pytest.approx(obj_gpu, rel=1e-6)
    return tie_all, tot


@pytest.mark.parametrize("c", [2, 3, 4])
def test_config_certificate_full(c):
    _check(_run(c))


def test_config5_certificate_sampled_rows():
    r = _run(5)
    m = r["cfg"].m
    _check(r, rows=[np.arange(256), np.arange(m // 2, m // 2 + 256), np.arange(m - 64, m)])
