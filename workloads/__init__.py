"""Seeded synthetic inputs for the BaKron solver: weights W and raw Gram factors.

This module is shared by the oracle side (``oracle/``, the tests) and the CUDA
side (the binding, ``bench.py``).  It holds no arithmetic of the method itself:
no damping, no Cholesky, no quantisation grid, no rounding.  It only draws
random matrices with the shapes and statistics of the paper's workload, which
is LLM linear layers calibrated on 256 sequences of 2048 tokens (Sec. 3.5
footnote; Appendix "Experiments"), with Kronecker factors built as Gram
matrices of activations / output-side vectors (Sec. 4.2, K-FAC style).

Recipe (every config):
  * Q_d: a random orthogonal d x d basis, QR of a standard-normal matrix with
    the sign of diag(R) folded into Q.  Without it the Grams would be diagonal,
    the unit-lower factors the identity and the solve plain round-to-nearest.
  * lambda_k = k^-alpha (k = 1..d); X = Q_d diag(sqrt(lambda)) Z, Z ~ N(0,1)
    of size d x N; Gram = X X^T / N.  alpha = 1 for the input side A, 0.5 for
    the output side B.
  * W: Gaussian (optionally with outlier columns) or Student-t, see CONFIGS.
Sub-seeds are 1000*c + {0: W, 1: Q_A, 2: Z_A, 3: Q_B, 4: Z_B, 5: outliers}.
Values depend on the torch device that draws them (CPU and CUDA generators
differ); each test or bench run draws once and hands the same bytes to both
sides.
"""
from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Config:
    index: int          # 1-based config number
    name: str
    m: int              # output features (rows of W, side of B)
    n: int              # input features (columns of W, side of A)
    n_samples: int      # calibration samples N behind each Gram
    w_dist: str         # "normal" | "normal_outliers" | "student_t"
    w_std: float
    w_dtype: torch.dtype
    bits: int
    group: int          # 0 = one grid per row, else columns per group
    damp: float = 0.01
    alpha_a: float = 1.0
    alpha_b: float = 0.5


CONFIGS = {
    1: Config(1, "single layer 128x128", 128, 128, 2048, "normal", 0.02,
              torch.float32, 4, 0),
    2: Config(2, "attention projection 4096x4096", 4096, 4096, 8192,
              "normal_outliers", 0.02, torch.bfloat16, 4, 0),
    3: Config(3, "MLP up-projection 11008x4096", 11008, 4096, 16384,
              "normal", 0.02, torch.bfloat16, 3, 0),
    4: Config(4, "MLP down-projection 4096x11008 g128", 4096, 11008, 16384,
              "student_t", 0.015, torch.bfloat16, 4, 128),
    5: Config(5, "70B-class MLP 28672x8192", 28672, 8192, 32768, "normal",
              0.01, torch.bfloat16, 2, 0),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def random_orthogonal(d: int, seed: int, device="cpu") -> torch.Tensor:
    """Haar-like orthogonal d x d matrix (fp32) from the QR of a Gaussian."""
    z = torch.randn(d, d, generator=_gen(seed, device), device=device,
                    dtype=torch.float32)
    q, r = torch.linalg.qr(z)
    return q * torch.sign(torch.diagonal(r))[None, :]


def power_law_gram(d: int, n_samples: int, alpha: float, seed_q: int,
                   seed_z: int, device="cpu", chunk: int = 8192) -> torch.Tensor:
    """Gram X X^T / N of N Gaussian samples with covariance Q diag(k^-alpha) Q^T.

    Accumulated in fp32 with TF32 disabled, in sample chunks so that X is never
    held whole.  The result is symmetrised exactly.
    """
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        q = random_orthogonal(d, seed_q, device)
        lam = torch.arange(1, d + 1, device=device, dtype=torch.float32)
        basis = q * lam.pow(-alpha / 2.0)[None, :]
        g = _gen(seed_z, device)
        gram = torch.zeros(d, d, device=device, dtype=torch.float32)
        done = 0
        while done < n_samples:
            k = min(chunk, n_samples - done)
            z = torch.randn(d, k, generator=g, device=device, dtype=torch.float32)
            x = basis @ z
            gram.addmm_(x, x.T)
            done += k
        gram /= float(n_samples)
        return 0.5 * (gram + gram.T)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev


def weights(cfg: Config, device="cpu") -> torch.Tensor:
    """W (m x n) in the config's storage dtype, per the config's distribution."""
    c = cfg.index
    g = _gen(1000 * c + 0, device)
    m, n = cfg.m, cfg.n
    if cfg.w_dist == "student_t":
        nu = 4.0
        z = torch.randn(m, n, generator=g, device=device, dtype=torch.float32)
        # chi-square with nu degrees of freedom as a sum of nu squared normals
        chi = torch.zeros(m, n, device=device, dtype=torch.float32)
        for _ in range(int(nu)):
            chi += torch.randn(m, n, generator=g, device=device,
                               dtype=torch.float32).square()
        t = z / torch.sqrt(chi / nu)
        w = t * (cfg.w_std / math.sqrt(nu / (nu - 2.0)))
    else:
        w = cfg.w_std * torch.randn(m, n, generator=g, device=device,
                                    dtype=torch.float32)
        if cfg.w_dist == "normal_outliers":
            k = max(1, round(0.001 * n))
            cols = torch.randperm(n, generator=_gen(1000 * c + 5, device),
                                  device=device)[:k]
            w[:, cols] *= 10.0
    return w.to(cfg.w_dtype)


def make(cfg: Config | int, device="cpu"):
    """(W, A_raw, B_raw) for a config; A_raw and B_raw are undamped fp32 Grams."""
    if isinstance(cfg, int):
        cfg = CONFIGS[cfg]
    c = cfg.index
    w = weights(cfg, device)
    a = power_law_gram(cfg.n, cfg.n_samples, cfg.alpha_a, 1000 * c + 1,
                       1000 * c + 2, device)
    b = power_law_gram(cfg.m, cfg.n_samples, cfg.alpha_b, 1000 * c + 3,
                       1000 * c + 4, device)
    return w, a, b


def small_problem(m: int, n: int, seed: int, n_samples: int | None = None,
                  w_std: float = 0.02, device="cpu"):
    """A random (W fp32, A_raw, B_raw) of any shape with the same recipe."""
    ns = n_samples if n_samples is not None else 2 * max(m, n) + 16
    g = _gen(seed, device)
    w = w_std * torch.randn(m, n, generator=g, device=device, dtype=torch.float32)
    a = power_law_gram(n, ns, 1.0, seed + 1, seed + 2, device)
    b = power_law_gram(m, ns, 0.5, seed + 3, seed + 4, device)
    return w, a, b
