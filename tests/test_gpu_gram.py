"""GPU parity of the Kronecker-factor accumulation (Sec. 4, "Choosing the
Factorization"): bakron_gram (G <- beta G + alpha X^T diag(w) X on the
tensor cores), bakron_sample_sqnorms and the K-FAC / one-step Shampoo factors,
against the float64 oracle.

Tolerance, from the arithmetic: each product is exact (bf16 samples, kind::f16)
or formed from tf32 hi/lo parts with a relative error below 2^-21; at most 256
products are summed in place in the tensor core's fp32 accumulator (<= 256 *
2^-23 of their absolute sum, about 3e-5) and the groups in fp32 registers
(<= k/256 * 2^-24), so |G - G_ref| <= 2^-14 * sum_t |alpha w_t x_ti x_tj| +
2^-20 |beta G0| holds for the sample counts used here (k <= 8192).
"""
import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import paper_2608_06291_gb300 as P


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.build()
    P.lib()


def _samples(k, d, seed, dtype):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(k, d, generator=g) * torch.linspace(0.2, 3.0, d)   # uneven feature scales
    return x.to(dtype)


def _check(G_gpu, X64, w64, alpha, beta, G0):
    ref = O.gram(X64, w64, alpha, beta, G0)
    ax = np.abs(X64)
    wa = np.ones(len(X64)) if w64 is None else np.abs(w64)
    bound = 2.0 ** -14 * abs(alpha) * ((ax * wa[:, None]).T @ ax)
    if beta != 0.0:
        bound += 2.0 ** -20 * abs(beta) * np.abs(G0)
    Gn = G_gpu.cpu().numpy().astype(np.float64)
    err = np.abs(Gn - ref)
    assert np.all(err <= bound + 1e-30), float((err / (bound + 1e-30)).max())
    np.testing.assert_array_equal(Gn, Gn.T)          # mirrored, not recomputed


@pytest.mark.parametrize("k,d", [(1, 1), (31, 5), (1000, 100), (257, 128), (700, 300)])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("weighted", [False, True])
def test_gram_matches_oracle(k, d, dtype, weighted):
    X = _samples(k, d, 10 * k + d, dtype)
    w = torch.rand(k, generator=torch.Generator().manual_seed(k)) * 2 if weighted else None
    G = P.bakron_gram(X.cuda(), None if w is None else w.cuda(), alpha=1.0 / k)
    torch.cuda.synchronize()
    _check(G, X.double().numpy(), None if w is None else w.double().numpy(), 1.0 / k, 0.0, None)


@pytest.mark.parametrize("dtype,weighted", [(torch.float32, True), (torch.bfloat16, False)])
def test_gram_beta_and_chunks(dtype, weighted):
    """beta applies once, before the first chunk; many small chunks (a
    workspace sized for 64 samples: 64 of them on the tf32 path, 256 on the
    bf16 one, whose last chunk ends in a partial group of slots) give the
    one-chunk result to rounding."""
    k, d = 1000, 200
    X = _samples(k, d, 3, dtype).cuda()
    w = (torch.rand(k, generator=torch.Generator().manual_seed(1)) + 0.5).cuda() if weighted \
        else None
    G0 = torch.randn(d, d, generator=torch.Generator().manual_seed(2))
    G0 = (G0 + G0.T).cuda()
    G1 = G0.clone()
    P.bakron_gram(X, w, alpha=0.25, beta=-0.5, G=G1)
    G2 = G0.clone()
    ws = torch.empty(P.bakron_gram_workspace_bytes(d, 64, weighted), dtype=torch.uint8,
                     device="cuda")
    P.bakron_gram(X, w, alpha=0.25, beta=-0.5, G=G2, workspace=ws)
    torch.cuda.synchronize()
    for G in (G1, G2):
        _check(G, X.double().cpu().numpy(), None if w is None else w.double().cpu().numpy(),
               0.25, -0.5, G0.double().cpu().numpy())


def test_gram_strided_operands():
    """X with a row stride above d, G a view into a wider buffer: the
    entries outside the d x d view stay untouched."""
    k, d = 300, 130
    Xb = _samples(k, d + 20, 9, torch.bfloat16).cuda()
    X = Xb[:, 7:7 + d]
    Gb = torch.full((d, d + 11), 7.0, device="cuda")
    G = Gb[:, :d]
    P.bakron_gram(X, alpha=1.0, beta=0.0, G=G)
    torch.cuda.synchronize()
    assert torch.all(Gb[:, d:] == 7.0)
    _check(G, X.double().cpu().numpy(), None, 1.0, 0.0, None)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_sample_sqnorms(dtype):
    Y = _samples(333, 77, 4, dtype).cuda()
    s = P.bakron_sample_sqnorms(Y)
    torch.cuda.synchronize()
    np.testing.assert_allclose(s.cpu().numpy(), O.sample_sqnorms(Y.double().cpu().numpy()),
                               rtol=1e-5)


def test_kfac_and_shampoo_factors():
    k = 640
    a = _samples(k, 96, 5, torch.bfloat16).cuda()
    b = _samples(k, 160, 6, torch.bfloat16).cuda()
    a64, b64 = a.double().cpu().numpy(), b.double().cpu().numpy()
    Ak, Bk = P.kfac_factors(a, b)
    As, Bs = P.shampoo_factors(a, b)
    torch.cuda.synchronize()
    rAk, rBk = O.kfac_factors(a64, b64)
    rAs, rBs = O.shampoo_factors(a64, b64, 1)
    for G, R in ((Ak, rAk), (Bk, rBk), (As, rAs), (Bs, rBs)):
        Gn = G.cpu().numpy().astype(np.float64)
        assert np.abs(Gn - R).max() <= 1e-5 * np.abs(R).max()


def test_gram_attention_width_sampled():
    """d = 4096 features, 8192 bf16 samples (the 4096 x 4096 projection's
    input side): 2000 sampled entries against fp64 dot products."""
    k, d = 8192, 4096
    X = _samples(k, d, 77, torch.bfloat16).cuda()
    G = P.bakron_gram(X, alpha=1.0 / k)
    torch.cuda.synchronize()
    rng = np.random.default_rng(0)
    I = rng.integers(0, d, 2000)
    J = rng.integers(0, d, 2000)
    Xh = X.double().cpu().numpy()
    ref = np.einsum("ti,ti->i", Xh[:, I], Xh[:, J]) / k
    bnd = 2.0 ** -14 * np.einsum("ti,ti->i", np.abs(Xh[:, I]), np.abs(Xh[:, J])) / k
    got = G.cpu().numpy()[I, J].astype(np.float64)
    assert np.all(np.abs(got - ref) <= bnd)
    Gc = G.cpu()
    assert torch.equal(Gc, Gc.T)


def test_gram_bench_workload_sampled():
    """The bench's workload: 65536 bf16 rows of 4096 features in one chunk;
    500 sampled entries against fp64 dot products, and exact symmetry."""
    k, d = 65536, 4096
    g = torch.Generator(device="cuda").manual_seed(4096)
    X = (torch.randn(k, d, generator=g, device="cuda")
         * torch.linspace(0.2, 3.0, d, device="cuda")).to(torch.bfloat16)
    ws = torch.empty(P.bakron_gram_workspace_bytes(d, k, False), dtype=torch.uint8,
                     device="cuda")
    G = P.bakron_gram(X, alpha=1.0 / k, workspace=ws)
    torch.cuda.synchronize()
    rng = np.random.default_rng(1)
    I = rng.integers(0, d, 500)
    J = rng.integers(0, d, 500)
    XI = X[:, torch.from_numpy(I).cuda()].double().cpu().numpy()
    XJ = X[:, torch.from_numpy(J).cuda()].double().cpu().numpy()
    ref = np.einsum("ti,ti->i", XI, XJ) / k
    bnd = 2.0 ** -14 * np.einsum("ti,ti->i", np.abs(XI), np.abs(XJ)) / k
    got = G.cpu().numpy()[I, J].astype(np.float64)
    assert np.all(np.abs(got - ref) <= bnd)
    assert torch.equal(G, G.T)
