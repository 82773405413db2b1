"""Thin ctypes binding of libbakron.so (include/bakron.h), same names as the C ABI.

Only argument marshalling lives here: every step of the solve runs in the
library's CUDA kernels.  torch supplies device memory and the current stream.
If the library is missing this module raises; there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import buildlib as _build

OK, ERR_INVALID_ARG, ERR_NOT_SPD, ERR_CUDA, ERR_TIMEOUT, ERR_WORKSPACE, ERR_NONFINITE = range(7)
F32, BF16 = 0, 1

_lib = None


class BakronError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        detail = ""
        if status == ERR_CUDA and _lib is not None:
            code, name, where, line = last_cuda_error()
            if code:
                detail = f" [{name} at {where}:{line}]"
        super().__init__(f"{what}: {strerror(status)} (status {status}){detail}")


def library_path() -> str:
    return _build.LIB


def lib() -> ctypes.CDLL:
    """Load libbakron.so (built by ``build()``); raise if it is absent."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with "
                           "paper_2608_06291_gb300.build.build() (no CPU fallback exists)")
    L = ctypes.CDLL(path)
    vp, i32, i64, sz, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t, ctypes.c_float
    L.bakron_factors_bytes.argtypes = [i32, i32]
    L.bakron_factors_bytes.restype = sz
    L.bakron_workspace_bytes.argtypes = [i32, i32]
    L.bakron_workspace_bytes.restype = sz
    L.bakron_prepare.argtypes = [vp, vp, i32, i32, f32, vp, vp, sz, vp]
    L.bakron_prepare.restype = i32
    L.bakron_set_factors.argtypes = [vp, vp, vp, vp, i32, i32, vp, vp]
    L.bakron_set_factors.restype = i32
    L.bakron_get_factors.argtypes = [vp, i32, i32, vp, vp, vp, vp, vp]
    L.bakron_get_factors.restype = i32
    L.bakron_solve.argtypes = [vp, i32, i32, i32, i64, vp, i32, i32, vp, vp, vp, vp, vp, sz, i32, vp]
    L.bakron_solve.restype = i32
    L.bakron_solve_gptq.argtypes = [vp, i32, i32, i32, i64, vp, i32, i32, vp, vp, vp, vp, vp, sz,
                                    i32, vp]
    L.bakron_solve_gptq.restype = i32
    L.bakron_grid_symmetric.argtypes = [vp, i32, i32, i32, i64, i32, i32, i32, vp, vp, vp]
    L.bakron_grid_symmetric.restype = i32
    L.bakron_solve_with_grid.argtypes = [vp, i32, i32, i32, i64, vp, i32, i32, vp, vp, vp, vp,
                                         vp, sz, i32, vp]
    L.bakron_solve_with_grid.restype = i32
    L.bakron_gram_workspace_bytes.argtypes = [i32, i32, i32]
    L.bakron_gram_workspace_bytes.restype = sz
    L.bakron_gram.argtypes = [vp, i32, i32, i32, i64, vp, f32, f32, vp, i64, vp, sz, i32, vp]
    L.bakron_gram.restype = i32
    L.bakron_sample_sqnorms.argtypes = [vp, i32, i32, i32, i64, vp, vp]
    L.bakron_sample_sqnorms.restype = i32
    L.bakron_batched_workspace_bytes.argtypes = [i32, i32, i32]
    L.bakron_batched_workspace_bytes.restype = sz
    pp = ctypes.POINTER(vp)
    L.bakron_solve_batched.argtypes = [i32, pp, i32, i32, i32, i64, pp, i32, i32, pp, pp, pp,
                                       vp, sz, i32, i32, vp]
    L.bakron_solve_batched.restype = i32
    L.bakron_read_status_batched.argtypes = [vp, i32, i32, i32, vp]
    L.bakron_read_status_batched.restype = i32
    L.bakron_solve_noalloc.argtypes = [vp, i32, i32, i32, i64, vp, i32, i32, vp, vp, vp, vp, i32, vp]
    L.bakron_solve_noalloc.restype = i32
    L.bakron_read_status_noalloc.argtypes = [vp]
    L.bakron_read_status_noalloc.restype = i32
    L.bakron_read_status.argtypes = [vp, vp]
    L.bakron_read_status.restype = i32
    L.bakron_profile_enable.argtypes = [i32]
    L.bakron_profile_enable.restype = i32
    L.bakron_profile_collect.argtypes = [vp]
    L.bakron_profile_collect.restype = i32
    dp = ctypes.POINTER(ctypes.c_double)
    L.bakron_profile_launch_stamps.argtypes = [i32, ctypes.POINTER(i32), dp, dp, dp]
    L.bakron_profile_launch_stamps.restype = i32
    L.bakron_diag_leaf_chain.argtypes = [vp, i32, vp, vp, vp, vp, vp, ctypes.c_size_t,
                                         ctypes.POINTER(ctypes.c_double), vp]
    L.bakron_diag_leaf_chain.restype = i32
    L.bakron_profile_read.argtypes = [i32, ctypes.POINTER(i32), ctypes.POINTER(ctypes.c_double),
                                      ctypes.POINTER(ctypes.c_double)]
    L.bakron_profile_read.restype = i32
    L.bakron_last_launches.argtypes = []
    L.bakron_last_launches.restype = i32
    L.bakron_diag_gemm_tf32x3.argtypes = [vp, vp, vp, i32, i32, i32, vp, sz, vp]
    L.bakron_diag_gemm_tf32x3.restype = i32
    L.bakron_autotune.argtypes = [vp, i32, i32, i32, i64, vp, i32, i32, vp, vp, vp, vp, sz,
                                  ctypes.POINTER(i32), ctypes.POINTER(i32), ctypes.POINTER(i32),
                                  ctypes.POINTER(ctypes.c_float), vp]
    L.bakron_autotune.restype = i32
    L.bakron_get_tuning.argtypes = [i32, i32, ctypes.POINTER(i32), ctypes.POINTER(i32),
                                    ctypes.POINTER(i32)]
    L.bakron_get_tuning.restype = i32
    L.bakron_autotune_clear.argtypes = []
    L.bakron_autotune_clear.restype = None
    L.bakron_diag_mma_rate.argtypes = [i32, vp, sz, ctypes.POINTER(ctypes.c_double),
                                       ctypes.POINTER(ctypes.c_double), vp]
    L.bakron_diag_mma_rate.restype = i32
    L.bakron_strerror.argtypes = [i32]
    L.bakron_strerror.restype = ctypes.c_char_p
    L.bakron_last_cuda_error.argtypes = [ctypes.POINTER(ctypes.c_char_p),
                                         ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(i32)]
    L.bakron_last_cuda_error.restype = i32
    _lib = L
    return L


def strerror(status: int) -> str:
    return lib().bakron_strerror(int(status)).decode()


def bakron_last_cuda_error():
    """(code, name, source file, line) of the CUDA error behind the last
    ERR_CUDA this thread got from the library (code 0: none)."""
    name, where, line = ctypes.c_char_p(), ctypes.c_char_p(), ctypes.c_int32()
    code = lib().bakron_last_cuda_error(ctypes.byref(name), ctypes.byref(where), ctypes.byref(line))
    return (int(code), (name.value or b"").decode(), (where.value or b"").decode(), int(line.value))


last_cuda_error = bakron_last_cuda_error


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(rc, what):
    if rc != OK:
        raise BakronError(rc, what)


def factors_bytes(m: int, n: int) -> int:
    return int(lib().bakron_factors_bytes(m, n))


def workspace_bytes(m: int, n: int) -> int:
    return int(lib().bakron_workspace_bytes(m, n))


def alloc_workspace(m: int, n: int, device="cuda") -> torch.Tensor:
    return torch.empty(workspace_bytes(m, n), dtype=torch.uint8, device=device)


class Factors:
    """Opaque device factor buffer for an m x n problem."""

    def __init__(self, m: int, n: int, device="cuda"):
        self.m, self.n = m, n
        self.buf = torch.empty(factors_bytes(m, n), dtype=torch.uint8, device=device)


def _as_f32_square(t, d, name):
    if t.dtype != torch.float32 or t.dim() != 2 or tuple(t.shape) != (d, d) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA float32 {d}x{d} tensor")
    return t.contiguous()


def bakron_prepare(A, B, damp: float = 0.01, workspace=None, stream=None) -> Factors:
    n, m = A.shape[0], B.shape[0]
    A = _as_f32_square(A, n, "A")
    B = _as_f32_square(B, m, "B")
    f = Factors(m, n, A.device)
    ws = workspace if workspace is not None else alloc_workspace(m, n, A.device)
    rc = lib().bakron_prepare(_ptr(A), _ptr(B), m, n, float(damp), _ptr(f.buf), _ptr(ws),
                              ws.numel(), _stream(stream))
    _check(rc, "bakron_prepare")
    return f


def bakron_set_factors(LA, LB, rA=None, rB=None, stream=None) -> Factors:
    n, m = LA.shape[0], LB.shape[0]
    LA = _as_f32_square(LA, n, "LA")
    LB = _as_f32_square(LB, m, "LB")
    rA = None if rA is None else rA.contiguous().float()
    rB = None if rB is None else rB.contiguous().float()
    f = Factors(m, n, LA.device)
    rc = lib().bakron_set_factors(_ptr(LA), _ptr(LB), _ptr(rA), _ptr(rB), m, n, _ptr(f.buf),
                                  _stream(stream))
    _check(rc, "bakron_set_factors")
    return f


def bakron_get_factors(f: Factors, stream=None):
    dev = f.buf.device
    LA = torch.empty(f.n, f.n, dtype=torch.float32, device=dev)
    LB = torch.empty(f.m, f.m, dtype=torch.float32, device=dev)
    rA = torch.empty(f.n, dtype=torch.float32, device=dev)
    rB = torch.empty(f.m, dtype=torch.float32, device=dev)
    rc = lib().bakron_get_factors(_ptr(f.buf), f.m, f.n, _ptr(LA), _ptr(LB), _ptr(rA), _ptr(rB),
                                  _stream(stream))
    _check(rc, "bakron_get_factors")
    return LA, LB, rA, rB


def _w_dtype(W):
    if not W.is_cuda or W.dim() != 2 or W.stride(1) != 1:
        raise ValueError("W must be a 2-D CUDA tensor with unit column stride")
    if W.dtype == torch.float32:
        return F32
    if W.dtype == torch.bfloat16:
        return BF16
    raise ValueError("W must be float32 or bfloat16")


def bakron_solve(W, f: Factors, bits: int, group_size: int = 0, workspace=None,
                 prerounding: bool = False, sync: bool = True, out=None, stream=None):
    """Round W (CUDA fp32/bf16, unit column stride).  Returns (codes uint8,
    scales, zeros[, prerounding fp32])."""
    dt = _w_dtype(W)
    m, n = W.shape
    if (f.m, f.n) != (m, n):
        raise ValueError("factor buffer was built for a different shape")
    G = 1 if group_size == 0 else n // group_size
    dev = W.device
    if out is None:
        codes = torch.empty(m, n, dtype=torch.uint8, device=dev)
        scales = torch.empty(m, G, dtype=torch.float32, device=dev)
        zeros = torch.empty(m, G, dtype=torch.float32, device=dev)
        xpre = torch.empty(m, n, dtype=torch.float32, device=dev) if prerounding else None
    else:
        codes, scales, zeros, xpre = out
    ws = workspace if workspace is not None else alloc_workspace(m, n, dev)
    rc = lib().bakron_solve(_ptr(W), dt, m, n, W.stride(0), _ptr(f.buf), int(bits),
                            int(group_size), _ptr(codes), _ptr(scales), _ptr(zeros), _ptr(xpre),
                            _ptr(ws), ws.numel(), 1 if sync else 0, _stream(stream))
    _check(rc, "bakron_solve")
    return (codes, scales, zeros, xpre) if prerounding else (codes, scales, zeros)


def bakron_solve_gptq(W, f: Factors, bits: int, group_size: int = 0, workspace=None,
                      prerounding: bool = False, sync: bool = True, out=None, stream=None):
    """The solve with B = I (GPTQ on every row under L^A of `f`); arguments
    and results as bakron_solve, group_size 0 or a multiple of 32."""
    dt = _w_dtype(W)
    m, n = W.shape
    if (f.m, f.n) != (m, n):
        raise ValueError("factor buffer was built for a different shape")
    G = 1 if group_size == 0 else n // group_size
    dev = W.device
    if out is None:
        codes = torch.empty(m, n, dtype=torch.uint8, device=dev)
        scales = torch.empty(m, G, dtype=torch.float32, device=dev)
        zeros = torch.empty(m, G, dtype=torch.float32, device=dev)
        xpre = torch.empty(m, n, dtype=torch.float32, device=dev) if prerounding else None
    else:
        codes, scales, zeros, xpre = out
    ws = workspace if workspace is not None else alloc_workspace(m, n, dev)
    rc = lib().bakron_solve_gptq(_ptr(W), dt, m, n, W.stride(0), _ptr(f.buf), int(bits),
                                 int(group_size), _ptr(codes), _ptr(scales), _ptr(zeros),
                                 _ptr(xpre), _ptr(ws), ws.numel(), 1 if sync else 0,
                                 _stream(stream))
    _check(rc, "bakron_solve_gptq")
    return (codes, scales, zeros, xpre) if prerounding else (codes, scales, zeros)


def bakron_grid_symmetric(W, levels: int = 3, group_size: int = 0, shrink_steps: int = 50,
                          stream=None):
    """The paper's experimental grid: symmetric codes {-l..l} with the
    MSE-shrunk max-abs scale per row (or per (row, group)).  Returns (scales,
    zeros), m x G fp32, zeros = l; asynchronous on `stream`."""
    dt = _w_dtype(W)
    m, n = W.shape
    G = 1 if group_size == 0 else n // group_size
    scales = torch.empty(m, G, dtype=torch.float32, device=W.device)
    zeros = torch.empty(m, G, dtype=torch.float32, device=W.device)
    rc = lib().bakron_grid_symmetric(_ptr(W), dt, m, n, W.stride(0), int(levels),
                                     int(group_size), int(shrink_steps), _ptr(scales),
                                     _ptr(zeros), _stream(stream))
    _check(rc, "bakron_grid_symmetric")
    return scales, zeros


def bakron_solve_with_grid(W, f: Factors, scales, zeros, qmax: int, group_size: int = 0,
                           workspace=None, prerounding: bool = False, sync: bool = True,
                           stream=None):
    """Round W onto the caller's grid (codes 0..qmax, value s (c - z)).
    Returns codes uint8 [, prerounding fp32]."""
    dt = _w_dtype(W)
    m, n = W.shape
    if (f.m, f.n) != (m, n):
        raise ValueError("factor buffer was built for a different shape")
    G = 1 if group_size == 0 else n // group_size
    for t, name in ((scales, "scales"), (zeros, "zeros")):
        if (not t.is_cuda or t.dtype != torch.float32 or tuple(t.shape) != (m, G)
                or not t.is_contiguous()):
            raise ValueError(f"{name} must be a contiguous CUDA float32 tensor of shape {(m, G)}")
    dev = W.device
    codes = torch.empty(m, n, dtype=torch.uint8, device=dev)
    xpre = torch.empty(m, n, dtype=torch.float32, device=dev) if prerounding else None
    ws = workspace if workspace is not None else alloc_workspace(m, n, dev)
    rc = lib().bakron_solve_with_grid(_ptr(W), dt, m, n, W.stride(0), _ptr(f.buf), int(qmax),
                                      int(group_size), _ptr(scales), _ptr(zeros), _ptr(codes),
                                      _ptr(xpre), _ptr(ws), ws.numel(), 1 if sync else 0,
                                      _stream(stream))
    _check(rc, "bakron_solve_with_grid")
    return (codes, xpre) if prerounding else codes


def _rows_dtype(X, name):
    if not X.is_cuda or X.dim() != 2 or X.stride(1) != 1:
        raise ValueError(f"{name} must be a 2-D CUDA tensor with unit column stride")
    if X.dtype == torch.float32:
        return F32
    if X.dtype == torch.bfloat16:
        return BF16
    raise ValueError(f"{name} must be float32 or bfloat16")


def bakron_gram_workspace_bytes(d: int, k_chunk: int, weighted: bool = False) -> int:
    return int(lib().bakron_gram_workspace_bytes(int(d), int(k_chunk), 1 if weighted else 0))


def bakron_gram(X, w=None, alpha: float = 1.0, beta: float = 0.0, G=None, workspace=None,
                chunk: int = 8192, sync: bool = True, stream=None):
    """G <- beta G + alpha X^T diag(w) X for X (k samples x d, CUDA fp32/bf16).
    Returns G (d x d fp32); a new G (beta ignored) when G is None."""
    dt = _rows_dtype(X, "X")
    k, d = X.shape
    if w is not None and (not w.is_cuda or w.dtype != torch.float32 or w.numel() != k
                          or not w.is_contiguous()):
        raise ValueError("w must be a contiguous CUDA float32 vector of length k")
    if G is None:
        G = torch.empty(d, d, dtype=torch.float32, device=X.device)
        beta = 0.0
    elif (not G.is_cuda or G.dtype != torch.float32 or tuple(G.shape) != (d, d)
          or G.stride(1) != 1):
        raise ValueError("G must be a CUDA float32 d x d tensor with unit column stride")
    if workspace is None:
        nb = bakron_gram_workspace_bytes(d, min(k, chunk), w is not None)
        workspace = torch.empty(nb, dtype=torch.uint8, device=X.device)
    rc = lib().bakron_gram(_ptr(X), dt, k, d, X.stride(0), _ptr(w), float(alpha), float(beta),
                           _ptr(G), G.stride(0), _ptr(workspace), workspace.numel(),
                           1 if sync else 0, _stream(stream))
    _check(rc, "bakron_gram")
    return G


def bakron_sample_sqnorms(Y, stream=None):
    """|y_t|^2 per row of Y (k x d, CUDA fp32/bf16) -> k fp32."""
    dt = _rows_dtype(Y, "Y")
    k, d = Y.shape
    out = torch.empty(k, dtype=torch.float32, device=Y.device)
    rc = lib().bakron_sample_sqnorms(_ptr(Y), dt, k, d, Y.stride(0), _ptr(out), _stream(stream))
    _check(rc, "bakron_sample_sqnorms")
    return out


def kfac_factors(a, b, stream=None):
    """K-FAC: (E[a a^T], E[b b^T]) from paired samples a (k x n), b (k x m)."""
    k = a.shape[0]
    return (bakron_gram(a, alpha=1.0 / k, stream=stream),
            bakron_gram(b, alpha=1.0 / k, stream=stream))


def shampoo_factors(a, b, stream=None):
    """One Shampoo power-iteration step from identity:
    (E[|b|^2 a a^T], E[|a|^2 b b^T])."""
    k = a.shape[0]
    wa = bakron_sample_sqnorms(b, stream)
    wb = bakron_sample_sqnorms(a, stream)
    return (bakron_gram(a, wa, alpha=1.0 / k, stream=stream),
            bakron_gram(b, wb, alpha=1.0 / k, stream=stream))


def bakron_batched_workspace_bytes(m: int, n: int, streams: int) -> int:
    return int(lib().bakron_batched_workspace_bytes(int(m), int(n), int(streams)))


def _ptr_array(ts):
    arr = (ctypes.c_void_p * len(ts))()
    for i, t in enumerate(ts):
        arr[i] = t.data_ptr()
    return arr


def bakron_solve_batched(Ws, fs, bits: int, group_size: int = 0, streams: int = 32,
                         workspace=None, sync: bool = True, out=None, stream=None):
    """Solve the H problems (Ws[h], fs[h]) of one shape side by side on
    min(streams, H) lanes (default: one per problem, up to the library's 32;
    32 heads of 128 x 4096 took 3.06 ms on 32 lanes against 4.10 ms on 16 on
    GB300).  Returns [(codes, scales, zeros)] per problem."""
    H = len(Ws)
    if H < 1 or len(fs) != H:
        raise ValueError("need as many factor buffers as weight matrices (>= 1)")
    m, n = Ws[0].shape
    dt = _w_dtype(Ws[0])
    ldw = Ws[0].stride(0)
    for W, f in zip(Ws, fs):
        if _w_dtype(W) != dt or tuple(W.shape) != (m, n) or W.stride(0) != ldw:
            raise ValueError("every W must have the same shape, dtype and row stride")
        if (f.m, f.n) != (m, n):
            raise ValueError("factor buffer was built for a different shape")
    G = 1 if group_size == 0 else n // group_size
    dev = Ws[0].device
    if out is None:
        out = [(torch.empty(m, n, dtype=torch.uint8, device=dev),
                torch.empty(m, G, dtype=torch.float32, device=dev),
                torch.empty(m, G, dtype=torch.float32, device=dev)) for _ in range(H)]
    S = min(int(streams), H)
    if workspace is None:
        workspace = torch.empty(bakron_batched_workspace_bytes(m, n, S), dtype=torch.uint8,
                                device=dev)
    rc = lib().bakron_solve_batched(
        H, _ptr_array(Ws), dt, m, n, ldw, _ptr_array([f.buf for f in fs]), int(bits),
        int(group_size), _ptr_array([o[0] for o in out]), _ptr_array([o[1] for o in out]),
        _ptr_array([o[2] for o in out]), _ptr(workspace), workspace.numel(), S,
        1 if sync else 0, _stream(stream))
    _check(rc, "bakron_solve_batched")
    return out


def bakron_autotune(W, f: Factors, bits: int, group_size: int = 0, workspace=None,
                    stream=None) -> dict:
    """Time the candidate schedules of an m x n solve on W and remember the
    fastest for later solves of that shape.  Returns {"tc_min_band",
    "fused_max_band", "leaf_block", "ms"}.  Synchronous; overwrites scratch
    outputs only."""
    if not W.is_cuda or W.dim() != 2 or W.stride(1) != 1:
        raise ValueError("W must be a 2-D CUDA tensor with unit column stride")
    dt = {torch.float32: F32, torch.bfloat16: BF16}.get(W.dtype)
    if dt is None:
        raise ValueError("W must be float32 or bfloat16")
    m, n = W.shape
    if (f.m, f.n) != (m, n):
        raise ValueError("factor buffer was built for a different shape")
    G = 1 if group_size == 0 else n // group_size
    dev = W.device
    codes = torch.empty(m, n, dtype=torch.uint8, device=dev)
    scales = torch.empty(m, G, dtype=torch.float32, device=dev)
    zeros = torch.empty(m, G, dtype=torch.float32, device=dev)
    ws = workspace if workspace is not None else alloc_workspace(m, n, dev)
    tc, fu, lb, ms = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0), ctypes.c_float(0.0)
    rc = lib().bakron_autotune(_ptr(W), dt, m, n, W.stride(0), _ptr(f.buf), int(bits),
                               int(group_size), _ptr(codes), _ptr(scales), _ptr(zeros), _ptr(ws),
                               ws.numel(), ctypes.byref(tc), ctypes.byref(fu), ctypes.byref(lb),
                               ctypes.byref(ms), _stream(stream))
    _check(rc, "bakron_autotune")
    return {"tc_min_band": tc.value, "fused_max_band": fu.value, "leaf_block": lb.value,
            "ms": ms.value}


def bakron_get_tuning(m: int, n: int) -> dict:
    """The schedule settings an m x n solve would use now."""
    tc, fu, lb = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0)
    _check(lib().bakron_get_tuning(int(m), int(n), ctypes.byref(tc), ctypes.byref(fu),
                                   ctypes.byref(lb)), "bakron_get_tuning")
    return {"tc_min_band": tc.value, "fused_max_band": fu.value, "leaf_block": lb.value}


def bakron_autotune_clear() -> None:
    lib().bakron_autotune_clear()


def bakron_solve_noalloc(W, f: Factors, bits: int, group_size: int = 0,
                         prerounding: bool = False, sync: bool = True, out=None, stream=None):
    """bakron_solve without a workspace argument, for callers that cannot
    allocate device scratch: the library's fixed 64 MiB array is used instead
    (problems whose solve scratch, about 20 * mp * np bytes, fits).  Outputs are
    allocated here unless ``out`` is given."""
    if not W.is_cuda or W.dim() != 2 or W.stride(1) != 1:
        raise ValueError("W must be a 2-D CUDA tensor with unit column stride")
    dt = {torch.float32: F32, torch.bfloat16: BF16}.get(W.dtype)
    if dt is None:
        raise ValueError("W must be float32 or bfloat16")
    m, n = W.shape
    if (f.m, f.n) != (m, n):
        raise ValueError("factor buffer was built for a different shape")
    G = 1 if group_size == 0 else n // group_size
    dev = W.device
    if out is None:
        codes = torch.empty(m, n, dtype=torch.uint8, device=dev)
        scales = torch.empty(m, G, dtype=torch.float32, device=dev)
        zeros = torch.empty(m, G, dtype=torch.float32, device=dev)
        xpre = torch.empty(m, n, dtype=torch.float32, device=dev) if prerounding else None
    else:
        codes, scales, zeros, xpre = out
    rc = lib().bakron_solve_noalloc(_ptr(W), dt, m, n, W.stride(0), _ptr(f.buf), int(bits),
                                    int(group_size), _ptr(codes), _ptr(scales), _ptr(zeros),
                                    _ptr(xpre), 1 if sync else 0, _stream(stream))
    _check(rc, "bakron_solve_noalloc")
    return (codes, scales, zeros, xpre) if prerounding else (codes, scales, zeros)


def bakron_read_status(workspace, stream=None) -> int:
    return int(lib().bakron_read_status(_ptr(workspace), _stream(stream)))


def bakron_read_status_noalloc(stream=None) -> int:
    """Status of the last bakron_solve_noalloc on the current device (read
    and cleared); the one way to see a device error of a sync=False call."""
    return int(lib().bakron_read_status_noalloc(_stream(stream)))


PROFILE_FAMILIES = ("init", "leaf", "band1", "band2", "copy", "tc1", "tc2", "fused", "subtree")


def bakron_profile_enable(on=True) -> None:
    """on: False (off), True or 1 (event mode), 2 (timeline mode)."""
    mode = 2 if on == 2 else (1 if on else 0)
    _check(lib().bakron_profile_enable(mode), "bakron_profile_enable")


def bakron_profile_collect(stream=None) -> None:
    """Timeline mode: fold the stamps of the last run of the recorded solve
    (e.g. one graph replay) into the family totals."""
    _check(lib().bakron_profile_collect(_stream(stream)), "bakron_profile_collect")


def bakron_profile_timeline() -> tuple:
    """Timeline mode: (runs collected, summed span of those runs in ms)."""
    n, ms = ctypes.c_int(0), ctypes.c_double(0.0)
    _check(lib().bakron_profile_read(-1, ctypes.byref(n), ctypes.byref(ms), None),
           "bakron_profile_read")
    return n.value, ms.value


def bakron_profile_launch_stamps(max_launches: int = 1 << 15) -> list:
    """Timeline mode: [(family name, flops, start_us, end_us)] of the last
    collected run, in enqueue order."""
    n = max_launches
    fam = (ctypes.c_int * n)()
    fl, st, en = (ctypes.c_double * n)(), (ctypes.c_double * n)(), (ctypes.c_double * n)()
    k = lib().bakron_profile_launch_stamps(n, fam, fl, st, en)
    if k < 0:
        _check(-k, "bakron_profile_launch_stamps")
    return [(PROFILE_FAMILIES[fam[i]], fl[i], st[i], en[i]) for i in range(min(k, n))]


def bakron_profile_read() -> dict:
    """{family: (launches, milliseconds, flops)} accumulated since the last enable."""
    out = {}
    for i, name in enumerate(PROFILE_FAMILIES):
        n = ctypes.c_int(0)
        ms = ctypes.c_double(0.0)
        fl = ctypes.c_double(0.0)
        _check(lib().bakron_profile_read(i, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(fl)),
               "bakron_profile_read")
        out[name] = (n.value, ms.value, fl.value)
    return out


def bakron_diag_leaf_chain(seed: int = 0, device=None) -> float:
    """Cycles of one step of the leaf's dependent chain, one tile alone on the
    GPU (a random 32 x 32 problem with identity factors)."""
    dev = device or torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(seed)
    W = 0.02 * torch.randn(32, 32, generator=g, device=dev)
    f = bakron_set_factors(torch.eye(32, device=dev), torch.eye(32, device=dev))
    codes = torch.empty(32, 32, dtype=torch.uint8, device=dev)
    sz = torch.empty(2, 32, 1, dtype=torch.float32, device=dev)
    ws = torch.empty(workspace_bytes(32, 32) + 256, dtype=torch.uint8, device=dev)
    cyc = ctypes.c_double(0.0)
    _check(lib().bakron_diag_leaf_chain(_ptr(W), F32, _ptr(f.buf), _ptr(codes), _ptr(sz[0]),
                                        _ptr(sz[1]), _ptr(ws), ws.numel(), ctypes.byref(cyc),
                                        _stream(None)), "bakron_diag_leaf_chain")
    return cyc.value


def bakron_last_launches() -> int:
    return int(lib().bakron_last_launches())


def bakron_diag_gemm_tf32x3(A, B, stream=None):
    """C = A B^T on the tensor cores with the solve's 3xTF32 split (diagnostic)."""
    A = A.contiguous()
    B = B.contiguous()
    M, K = A.shape
    N = B.shape[0]
    C = torch.empty(M, N, dtype=torch.float32, device=A.device)
    ws = torch.empty(256 + 8 * (M + N) * K, dtype=torch.uint8, device=A.device)
    rc = lib().bakron_diag_gemm_tf32x3(_ptr(A), _ptr(B), _ptr(C), M, N, K, _ptr(ws), ws.numel(),
                                       _stream(stream))
    _check(rc, "bakron_diag_gemm_tf32x3")
    return C


def dequantize(codes, scales, zeros):
    """Values s * (c - z) of a code matrix (a convenience for callers)."""
    m, n = codes.shape
    g = n // scales.shape[1]
    s = scales.repeat_interleave(g, dim=1)
    z = zeros.repeat_interleave(g, dim=1)
    return s * (codes.float() - z)


def bakron_diag_mma_rate(stages: int = 2000, stream=None) -> dict:
    """Measured tcgen05 kind::tf32 MMA rate of the whole device (diagnostic).
    Returns {"tf32_tflops", "cycles_per_mma", "fp32_effective_tflops"}."""
    ws = torch.empty(256 + 8 * 1024, dtype=torch.uint8, device="cuda")
    tf, cyc = ctypes.c_double(0.0), ctypes.c_double(0.0)
    _check(lib().bakron_diag_mma_rate(int(stages), _ptr(ws), ws.numel(), ctypes.byref(tf),
                                      ctypes.byref(cyc), _stream(stream)),
           "bakron_diag_mma_rate")
    return {"tf32_tflops": tf.value, "cycles_per_mma": cyc.value,
            "fp32_effective_tflops": tf.value / 3.0}
