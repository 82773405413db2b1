"""The C ABI without a GPU: every declared symbol is exported, sizes are sane,
and invalid arguments are rejected on the host before any CUDA call."""
import ctypes
import os
import re

import pytest
import torch

import paper_2608_06291_gb300 as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            src = open(os.path.join(ROOT, "include", h)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(bakron_\w+)\s*\(", src))
    return names


@pytest.fixture(scope="module")
def L():
    P.build()
    return P.lib()


def test_every_declared_symbol_is_exported(L):
    names = declared_symbols()
    assert {"bakron_prepare", "bakron_solve", "bakron_factors_bytes"} <= names
    for name in sorted(names):
        assert hasattr(L, name), name


def test_sizes(L):
    assert P.factors_bytes(0, 5) == 0 and P.workspace_bytes(5, 0) == 0
    small = P.workspace_bytes(1, 1)
    assert small > 0
    # 128 x 128 padding: three fp32 planes at least
    assert P.workspace_bytes(4096, 4096) >= 3 * 4096 * 4096 * 4
    assert P.factors_bytes(4096, 4096) >= 2 * 4096 * 4096 * 4
    assert P.factors_bytes(100, 200) == P.factors_bytes(128, 256)


def test_invalid_arguments_rejected_on_host(L):
    vp = ctypes.c_void_p
    fake = vp(0x1000)  # never dereferenced: validation fails first
    # null W
    assert L.bakron_solve(None, 0, 4, 4, 4, fake, 4, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    # bad bits / dtype / group / ldw / shape
    assert L.bakron_solve(fake, 0, 4, 4, 4, fake, 9, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert L.bakron_solve(fake, 7, 4, 4, 4, fake, 4, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert L.bakron_solve(fake, 0, 4, 6, 6, fake, 4, 4, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert L.bakron_solve(fake, 0, 4, 6, 5, fake, 4, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert L.bakron_solve(fake, 0, 0, 6, 6, fake, 4, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    # workspace too small
    assert L.bakron_solve(fake, 0, 4, 4, 4, fake, 4, 0, fake, fake, fake, None, fake, 16, 0, None) == 5
    assert L.bakron_prepare(fake, fake, 4, 4, ctypes.c_float(-1.0), fake, fake, 1 << 30, None) == 1
    assert L.bakron_prepare(fake, fake, 4, 4, ctypes.c_float(0.01), fake, fake, 16, None) == 5
    assert L.bakron_set_factors(None, fake, None, None, 4, 4, fake, None) == 1
    assert L.bakron_read_status(None, None) == 1
    # no-alloc solve: sides beyond 131072 are invalid (as for bakron_solve);
    # valid problems whose scratch exceeds the fixed 64 MiB are refused as
    # a workspace shortfall -- both on the host, before any device call
    na = L.bakron_solve_noalloc
    assert na(fake, 0, (1 << 17) + 1, 4, 4, fake, 4, 0, fake, fake, fake, None, 1, None) == 1
    assert na(fake, 0, 4, (1 << 17) + 1, (1 << 17) + 1, fake, 4, 0, fake, fake, fake, None, 1,
              None) == 1
    assert na(fake, 0, 4096, 4096, 4096, fake, 4, 0, fake, fake, fake, None, 1, None) == 5
    assert na(fake, 0, 1792, 1793, 1793, fake, 4, 0, fake, fake, fake, None, 1, None) == 5
    assert na(None, 0, 4, 4, 4, fake, 4, 0, fake, fake, fake, None, 1, None) == 1
    # symmetric grid: levels, shrink steps, group, ldw, dtype
    g = L.bakron_grid_symmetric
    assert g(None, 0, 4, 4, 4, 3, 0, 50, fake, fake, None) == 1
    assert g(fake, 0, 4, 4, 4, 0, 0, 50, fake, fake, None) == 1
    assert g(fake, 0, 4, 4, 4, 128, 0, 50, fake, fake, None) == 1
    assert g(fake, 0, 4, 4, 4, 3, 0, -1, fake, fake, None) == 1
    assert g(fake, 0, 4, 4, 4, 3, 0, 1025, fake, fake, None) == 1
    assert g(fake, 0, 4, 6, 6, 3, 4, 50, fake, fake, None) == 1
    assert g(fake, 0, 4, 6, 5, 3, 0, 50, fake, fake, None) == 1
    assert g(fake, 2, 4, 4, 4, 3, 0, 50, fake, fake, None) == 1
    # solve with the caller's grid: qmax, null grid, group, workspace
    sg = L.bakron_solve_with_grid
    assert sg(fake, 0, 4, 4, 4, fake, 0, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert sg(fake, 0, 4, 4, 4, fake, 256, 0, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert sg(fake, 0, 4, 4, 4, fake, 6, 0, None, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert sg(fake, 0, 4, 6, 6, fake, 6, 4, fake, fake, fake, None, fake, 1 << 30, 0, None) == 1
    assert sg(fake, 0, 4, 4, 4, fake, 6, 0, fake, fake, fake, None, fake, 16, 0, None) == 5
    # Gram accumulation: k, d, strides, dtype, workspace
    gr = L.bakron_gram
    f1, f0 = ctypes.c_float(1.0), ctypes.c_float(0.0)
    assert gr(None, 0, 8, 4, 4, None, f1, f0, fake, 4, fake, 1 << 30, 0, None) == 1
    assert gr(fake, 0, 0, 4, 4, None, f1, f0, fake, 4, fake, 1 << 30, 0, None) == 1
    assert gr(fake, 0, 8, 4, 3, None, f1, f0, fake, 4, fake, 1 << 30, 0, None) == 1
    assert gr(fake, 0, 8, 4, 4, None, f1, f0, fake, 3, fake, 1 << 30, 0, None) == 1
    assert gr(fake, 0, 8, (1 << 16) + 1, 1 << 17, None, f1, f0, fake, 1 << 17, fake, 1 << 40,
              0, None) == 1
    assert gr(fake, 3, 8, 4, 4, None, f1, f0, fake, 4, fake, 1 << 30, 0, None) == 1
    need = L.bakron_gram_workspace_bytes(4, 1, 0)
    assert need == 256 + 2 * 128 * 32 * 4
    assert L.bakron_gram_workspace_bytes(4, 33, 1) == 256 + 4 * 128 * 64 * 4
    assert L.bakron_gram_workspace_bytes(0, 1, 0) == 0
    assert gr(fake, 0, 8, 4, 4, None, f1, f0, fake, 4, fake, need - 1, 0, None) == 5
    assert gr(fake, 0, 8, 4, 4, fake, f1, f0, fake, 4, fake, need, 0, None) == 5   # weighted: 4 planes
    # batched solve: H, lanes, null pointer arrays / entries, workspace
    pp = ctypes.c_void_p * 2
    arr, bad = pp(0x1000, 0x2000), pp(0x1000, None)
    b = L.bakron_solve_batched
    assert b(0, arr, 0, 4, 4, 4, arr, 4, 0, arr, arr, arr, fake, 1 << 30, 2, 0, None) == 1
    assert b(2, arr, 0, 4, 4, 4, arr, 4, 0, arr, arr, arr, fake, 1 << 30, 0, 0, None) == 1
    assert b(2, arr, 0, 4, 4, 4, arr, 4, 0, arr, arr, arr, fake, 1 << 30, 33, 0, None) == 1
    assert b(2, None, 0, 4, 4, 4, arr, 4, 0, arr, arr, arr, fake, 1 << 30, 2, 0, None) == 1
    assert b(2, arr, 0, 4, 4, 4, bad, 4, 0, arr, arr, arr, fake, 1 << 30, 2, 0, None) == 1
    assert b(2, arr, 0, 4, 4, 4, arr, 9, 0, arr, arr, arr, fake, 1 << 30, 2, 0, None) == 1
    one = L.bakron_batched_workspace_bytes(4, 4, 1)
    assert one > 0 and one % 256 == 0          # the solve's scratch alone
    assert L.bakron_batched_workspace_bytes(4, 4, 3) == 3 * one
    assert L.bakron_batched_workspace_bytes(4, 4, 0) == 0
    assert b(2, arr, 0, 4, 4, 4, arr, 4, 0, arr, arr, arr, fake, 2 * one - 1, 2, 0, None) == 5
    # with H = 1 only one lane is needed
    assert b(1, arr, 0, 4, 4, 4, arr, 4, 0, arr, arr, arr, fake, one - 1, 8, 0, None) == 5
    sq = L.bakron_sample_sqnorms
    assert sq(None, 0, 4, 4, 4, fake, None) == 1
    assert sq(fake, 0, 4, 4, 3, fake, None) == 1
    assert sq(fake, 0, 0, 4, 4, fake, None) == 1
    assert P.strerror(2) == "damped Gram is not positive definite"


@pytest.mark.skipif(torch.cuda.is_available(), reason="needs a machine without a CUDA device")
def test_cuda_failure_is_recorded_with_its_name_and_place(L):
    """A CUDA runtime failure surfaces as BAKRON_ERR_CUDA, and the error
    behind it (here: no device) can be read back with where it happened."""
    fake = ctypes.c_void_p(4096)
    assert L.bakron_read_status(fake, None) == 3
    code, name, where, line = P.bakron_last_cuda_error()
    assert code != 0 and name.startswith("cuda") and where == "capi.cu" and line > 0
    with pytest.raises(P.BakronError, match=r"\[cuda\w+ at capi\.cu:\d+\]"):
        P.bakron.__dict__["_check"](3, "probe")


def test_binding_rejects_bad_tensors_before_the_library():
    """The ctypes binding checks device, dtype and shapes itself and raises
    ValueError before calling into the library (no GPU needed)."""
    cpu = torch.zeros(8, 4)
    with pytest.raises(ValueError):
        P.bakron_gram(cpu)                               # not a CUDA tensor
    with pytest.raises(ValueError):
        P.bakron_sample_sqnorms(cpu)
    with pytest.raises(ValueError):
        P.bakron_grid_symmetric(cpu)
    with pytest.raises(ValueError):
        P.bakron_solve_batched([], [], 4)                # no problems
    with pytest.raises(ValueError):
        P.bakron_solve_batched([cpu], [], 4)             # factors missing


def test_header_is_plain_c(tmp_path):
    """include/bakron.h compiles as C99 (-pedantic, warnings as errors): the
    boundary carries no C++ or CUDA types."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    src = tmp_path / "use.c"
    src.write_text('#include "bakron.h"\nint main(void) { return bakron_strerror(0) == 0; }\n')
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", inc,
                        "-c", str(src), "-o", str(tmp_path / "use.o")],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
