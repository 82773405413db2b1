"""bakron_solve_noalloc against bakron_solve, through the C ABI.

The no-alloc entry point serves callers that cannot allocate device memory of
their own (a plugin handed only its input and output buffers by a framework
that owns every allocation, or a process under a fixed device-memory budget):
it runs the same solve with the library's fixed 64 MiB scratch array instead of
a caller workspace.  Two calls in a row, on different problems, must each give
the codes, grid and pre-rounding values of bakron_solve on the same inputs
(within the tests' 1e-4 grid-unit tolerance; in practice bit-identical); a
problem larger than the fixed scratch must be refused before any work, and
the largest square problem that fits must run; a device error of an
asynchronous call must be readable afterwards.
"""
import pytest
import torch

import workloads as WL

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


def _problem(m, n, seed, bits, group):
    W, A, B = WL.small_problem(m, n, seed, device="cuda")
    fac = P.bakron_prepare(A, B, 0.01)
    return W, fac, bits, group


def _same_solve(W, fac, bits, group):
    want = P.bakron_solve(W, fac, bits, group, prerounding=True)
    got = P.bakron_solve_noalloc(W, fac, bits, group, prerounding=True)
    torch.cuda.synchronize()
    assert torch.equal(got[0], want[0])                # codes
    assert torch.equal(got[1], want[1]) and torch.equal(got[2], want[2])
    s = want[1].repeat_interleave(W.shape[1] // want[1].shape[1], dim=1)
    dx = ((got[3] - want[3]).abs() / s).max().item()
    assert dx < 1e-4


def test_noalloc_matches_solve_on_two_calls_in_a_row():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    problems = [_problem(300, 417, 71, 4, 0), _problem(520, 256, 72, 3, 64)]
    for W, fac, bits, group in problems:
        _same_solve(W, fac, bits, group)


def test_noalloc_scratch_limit():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    L = P.lib()
    t = torch.zeros(16, dtype=torch.uint8, device="cuda")
    p = t.data_ptr()
    # 4096 x 4096 needs more than 20 * 4096^2 bytes > 64 MiB: refused on the host
    rc = L.bakron_solve_noalloc(p, 0, 4096, 4096, 4096, p, 4, 0, p, p, p, None, 1, None)
    assert rc == 5
    assert P.strerror(rc) == "workspace too small"
    # 1792 x 1792 (20 * 1792^2 bytes plus the tile flags and counters) fits and
    # runs; one more column pads n to 1920 and no longer fits
    W, fac, bits, group = _problem(1792, 1792, 73, 4, 0)
    _same_solve(W, fac, bits, group)
    rc = L.bakron_solve_noalloc(p, 0, 1792, 1793, 1793, p, 4, 0, p, p, p, None, 1, None)
    assert rc == 5


def test_noalloc_async_status_is_readable():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    fac = P.bakron_set_factors(torch.eye(40, device="cuda"), torch.eye(8, device="cuda"))
    W = torch.randn(8, 40, device="cuda")
    W[3, 7] = float("nan")
    P.bakron_solve_noalloc(W, fac, 4, sync=False)      # returns after enqueueing
    assert P.bakron_read_status_noalloc() == 6          # BAKRON_ERR_NONFINITE
    assert P.bakron_read_status_noalloc() == 0          # read clears it
    W[3, 7] = 0.0
    codes = P.bakron_solve_noalloc(W, fac, 4, sync=False)[0]
    assert P.bakron_read_status_noalloc() == 0
    want = P.bakron_solve(W, fac, 4)[0]
    assert torch.equal(codes, want)
