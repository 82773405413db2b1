"""The seeded input generators hold to the recipe stated for them: determinism,
orthogonal bases, power-law Gram spectra k^-alpha, exact symmetry, and the
weight distributions (Gaussian, outlier columns x10, Student-t rescaled to
the stated standard deviation)."""
import dataclasses
import math

import numpy as np
import torch

import workloads as WL


def test_same_seed_same_bytes():
    a = WL.make(1)
    b = WL.make(1)
    for x, y in zip(a, b):
        assert torch.equal(x, y)
    w1, _, _ = WL.small_problem(20, 30, 5)
    w2, _, _ = WL.small_problem(20, 30, 6)
    assert not torch.equal(w1, w2)


def test_config_shapes_and_dtypes():
    W, A, B = WL.make(1)
    cfg = WL.CONFIGS[1]
    assert W.shape == (cfg.m, cfg.n) and W.dtype == cfg.w_dtype
    assert A.shape == (cfg.n, cfg.n) and B.shape == (cfg.m, cfg.m)
    assert A.dtype == torch.float32 and B.dtype == torch.float32
    assert torch.equal(A, A.T) and torch.equal(B, B.T)
    # the configs of the recipe
    shapes = {c: (k.m, k.n, k.bits, k.group) for c, k in WL.CONFIGS.items()}
    assert shapes == {1: (128, 128, 4, 0), 2: (4096, 4096, 4, 0), 3: (11008, 4096, 3, 0),
                      4: (4096, 11008, 4, 128), 5: (28672, 8192, 2, 0)}


def test_orthogonal_basis():
    Q = WL.random_orthogonal(48, 3).double()
    np.testing.assert_allclose((Q.T @ Q).numpy(), np.eye(48), atol=1e-5)


def test_power_law_spectrum():
    """Eigenvalues of X X^T / N follow k^-alpha: the log-log slope of the
    spectrum is -alpha within sampling error (d = 64, N = 16384)."""
    for alpha in (1.0, 0.5):
        G = WL.power_law_gram(64, 16384, alpha, 11, 12).double().numpy()
        ev = np.sort(np.linalg.eigvalsh(G))[::-1]
        k = np.arange(1, 65)
        slope = np.polyfit(np.log(k), np.log(ev), 1)[0]
        assert abs(slope + alpha) < 0.08, (alpha, slope)
        np.testing.assert_allclose(ev[:8], k[:8] ** -alpha, rtol=0.1)


def _small(cfg_index, dist, m=256, n=2000, std=0.02):
    return dataclasses.replace(WL.CONFIGS[2], index=cfg_index, m=m, n=n, w_dist=dist,
                               w_std=std, w_dtype=torch.float32)


def test_weight_distributions():
    g = WL.weights(_small(91, "normal"))
    assert abs(float(g.std()) - 0.02) < 0.001
    t = WL.weights(_small(92, "student_t", std=0.015))
    assert abs(float(t.std()) - 0.015) < 0.0015          # rescaled to the stated std
    kurt = float(((t - t.mean()) ** 4).mean() / t.var() ** 2)
    assert kurt > 4.5                                      # heavy tails (Gaussian: 3)
    o = WL.weights(_small(93, "normal_outliers"))
    col_std = o.std(dim=0)
    big = int((col_std > 5 * 0.02).sum())
    assert big == max(1, round(0.001 * 2000))             # 0.1% of the columns, x10
    assert abs(float(col_std[col_std < 5 * 0.02].mean()) - 0.02) < 0.001
