"""GPU tests of bakron_solve_batched: H independent problems of one shape on
several lane streams give, problem by problem, the codes of bakron_solve
(bit for bit: the same kernels in the same order per problem) and agree with
the float64 oracle; the call can be captured into a CUDA graph.  With one
lane per problem the leaves of all problems share one launch per tile
anti-diagonal (the per-problem arithmetic is the same, so the codes are
still bit for bit those of bakron_solve).

The per-head setting (Sec. 4, local attention Hessians; BoA): W_Q of one
layer split into heads of 64 rows, a shared input-side A and one small
output-side B per head.
"""
import numpy as np
import pytest
import torch

import oracle as O
import workloads as WL
from tests._helpers import compare_codes, oracle_factors_fp32, to_np

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    P.lib()


def _heads(H, mh, n, seed):
    """W_Q rows split per head (bf16), A shared, one B per head."""
    W, A, _ = WL.small_problem(H * mh, n, seed)
    Bs = [WL.small_problem(mh, 8, seed + 100 + h)[2] for h in range(H)]
    return W, A, Bs


@pytest.mark.parametrize("streams,tc", [(1, False), (3, False), (8, False), (6, True), (2, True)])
def test_batched_equals_single_solves(streams, tc, monkeypatch):
    if tc:   # small leaf blocks and tensor cores on every node: band stages on each lane
        monkeypatch.setenv("BAKRON_LEAF_BLOCK", "4")
        monkeypatch.setenv("BAKRON_TC_MIN_BAND", "2")
        monkeypatch.setenv("BAKRON_SUBTREE_MAX", "0")
    H, mh, n = 6, 64, 200
    W, A, Bs = _heads(H, mh, n, 31)
    Wd = W.cuda().to(torch.bfloat16)
    Ws = [Wd[h * mh:(h + 1) * mh] for h in range(H)]             # row stride n
    fs = [P.bakron_prepare(A.cuda(), Bs[h].cuda(), 0.01) for h in range(H)]
    outs = P.bakron_solve_batched(Ws, fs, 4, 0, streams=streams)
    batched_launches = P.bakron_last_launches()   # the batched call's, before the checks below
    torch.cuda.synchronize()
    for h in range(H):
        c, s, z = P.bakron_solve(Ws[h], fs[h], 4, 0)
        assert torch.equal(outs[h][0], c)
        assert torch.equal(outs[h][1], s) and torch.equal(outs[h][2], z)
    assert batched_launches > H


def test_batched_matches_oracle_with_groups():
    H, mh, n = 4, 40, 160
    W, A, Bs = _heads(H, mh, n, 57)
    Ws, fs, refs = [], [], []
    for h in range(H):
        f, LA32, LB32 = oracle_factors_fp32(A, Bs[h], 0.01)
        fac = P.bakron_set_factors(torch.from_numpy(LA32).cuda(), torch.from_numpy(LB32).cuda())
        Wh = W[h * mh:(h + 1) * mh].contiguous()
        Ws.append(Wh.cuda())
        fs.append(fac)
        refs.append((to_np(Wh), LA32.astype(np.float64), LB32.astype(np.float64)))
    outs = P.bakron_solve_batched(Ws, fs, 3, 32, streams=4)
    torch.cuda.synchronize()
    for h in range(H):
        W64, LA, LB = refs[h]
        g = O.quant_grid(W64, 3, 32)
        np.testing.assert_array_equal(outs[h][1].cpu().numpy(), g.s)
        ref = O.bakron_recursive(W64, LA, LB, g)
        c = outs[h][0].cpu().numpy().astype(np.int64)
        st = compare_codes(W64, c, g, LA, LB, ref.codes)
        assert st["cert_mismatch_outside_band"] == 0, st
        if st["cert_mismatch"] == 0:
            np.testing.assert_array_equal(c, ref.codes)


@pytest.mark.parametrize("S", [3, 5])
def test_batched_graph_capture(S):
    """Captured once (after a first eager call created the lanes), replayed
    on new inputs: the results follow the inputs (S = 5: one lane per problem)."""
    H, mh, n = 5, 64, 256
    W, A, Bs = _heads(H, mh, n, 77)
    fs = [P.bakron_prepare(A.cuda(), Bs[h].cuda(), 0.01) for h in range(H)]
    Wd = W.cuda()
    Ws = [Wd[h * mh:(h + 1) * mh] for h in range(H)]
    ws = torch.empty(P.bakron_batched_workspace_bytes(mh, n, S), dtype=torch.uint8, device="cuda")
    outs = P.bakron_solve_batched(Ws, fs, 4, 0, streams=S, workspace=ws)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            P.bakron_solve_batched(Ws, fs, 4, 0, streams=S, workspace=ws, sync=False, out=outs,
                                   stream=s)
    Wd.mul_(-0.5)                      # new inputs in the captured buffers
    g.replay()
    torch.cuda.synchronize()
    assert P.lib().bakron_read_status_batched(ws.data_ptr(), mh, n, S, None) == 0
    for h in range(H):
        c, sc, z = P.bakron_solve(Ws[h], fs[h], 4, 0)
        assert torch.equal(outs[h][0], c) and torch.equal(outs[h][1], sc)


def test_batched_bench_workload_certificate():
    """The bench's workload: the 4096 x 4096 layer as 32 heads of 128 x 4096
    over 32 lanes (one per head), each head certified (teacher-forced, every
    entry) against fp64 factors of its own damped Grams."""
    cfg = WL.CONFIGS[2]
    W, A, _ = WL.make(cfg, device="cuda")
    Hh, mh, n = 32, 128, cfg.n
    Bs = [WL.power_law_gram(mh, cfg.n_samples, cfg.alpha_b, 9000 + h, 9100 + h, "cuda")
          for h in range(Hh)]
    LA, _, rA, _ = P.bakron_get_factors(P.bakron_prepare(A, Bs[0], cfg.damp))
    fs = []
    for h in range(Hh):
        LBh, _, rBh, _ = P.bakron_get_factors(P.bakron_prepare(Bs[h], Bs[h], cfg.damp))
        fs.append(P.bakron_set_factors(LA, LBh, rA, rBh))
    Ws = [W[h * mh:(h + 1) * mh] for h in range(Hh)]
    outs = P.bakron_solve_batched(Ws, fs, cfg.bits, 0, streams=32)
    torch.cuda.synchronize()
    RA = O.rev_cholesky(O.damped(to_np(A), cfg.damp))
    W64 = to_np(W.float())
    for h in range(Hh):
        RB = O.rev_cholesky(O.damped(to_np(Bs[h]), cfg.damp))
        Wh = W64[h * mh:(h + 1) * mh]
        g = O.quant_grid(Wh, cfg.bits, 0)
        np.testing.assert_array_equal(outs[h][1].cpu().numpy(), g.s)
        c = outs[h][0].cpu().numpy().astype(np.int64)
        rows = np.arange(mh)
        D = O.dequantize(c, g, n) - Wh
        _, bad, dist = O.certificate_rows(Wh, c, D, g, RA, RB, rows)
        assert int((bad & (dist >= 1e-4)).sum()) == 0, h
        assert int(bad.sum()) <= 1e-3 * bad.size
