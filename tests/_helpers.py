"""Shared test helpers: oracle runs on the exact inputs the GPU receives."""
import numpy as np
import torch

import oracle as O

TIE_BAND = 1e-4   # grid units: |x/s - (k + 1/2)| below this is a tie (the parity bar's tie rule)


def to_np(t):
    return t.detach().to("cpu", torch.float64).numpy()


def oracle_factors_fp32(A, B, damp):
    """Oracle factors rounded to fp32 (what the GPU solve receives) and the
    same values back in fp64 (what the oracle solves with)."""
    f = O.prepare(to_np(A), to_np(B), damp, via_inverse=False)
    LA32 = f.LA.astype(np.float32)
    LB32 = f.LB.astype(np.float32)
    return f, LA32, LB32


def compare_codes(W64, codes_gpu, g, LA64, LB64, ref_codes=None):
    """Teacher-forced certificate + raw match.  Returns a dict of statistics."""
    X, bad, dist = O.certificate(W64, codes_gpu, g, LA64, LB64)
    out = {"cert_mismatch": int(bad.sum()),
           "cert_mismatch_outside_band": int((bad & (dist >= TIE_BAND)).sum()),
           "n": codes_gpu.size, "X": X}
    if ref_codes is not None:
        out["raw_match"] = float((ref_codes == codes_gpu).mean())
    return out


def root_mismatches(bad: np.ndarray) -> np.ndarray:
    """Mismatches with no mismatch up-left of them (i <= p, j <= q, (i, j) !=
    (p, q)): the entries where two solves first part."""
    seen = np.maximum.accumulate(np.maximum.accumulate(bad, axis=0), axis=1)
    before = np.zeros_like(bad)
    before[1:, :] |= seen[:-1, :]
    before[:, 1:] |= seen[:, :-1]
    return bad & ~before
