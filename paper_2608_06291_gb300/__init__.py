"""GB300-native BaKron solver: two-sided Babai/GPTQ rounding under A (x) B.

The compute path is libbakron.so (hand-written sm_103a CUDA kernels behind the
C ABI in include/bakron.h); this package is its build script and a thin
ctypes binding with the same entry-point names.
"""
from .bakron import (BakronError, Factors, alloc_workspace, bakron_diag_gemm_tf32x3,  # noqa: F401
                     bakron_diag_mma_rate, bakron_diag_leaf_chain,
                     bakron_autotune, bakron_autotune_clear, bakron_get_factors,
                     bakron_get_tuning, bakron_grid_symmetric, bakron_solve_with_grid,
                     bakron_gram, bakron_gram_workspace_bytes, bakron_sample_sqnorms,
                     kfac_factors, shampoo_factors, bakron_solve_batched,
                     bakron_batched_workspace_bytes,
                     bakron_last_launches, bakron_prepare, bakron_profile_enable,
                     bakron_profile_read, bakron_profile_collect, bakron_profile_timeline,
                     bakron_profile_launch_stamps,
                     bakron_read_status, bakron_set_factors, bakron_solve, bakron_solve_gptq,
                     bakron_solve_noalloc, bakron_read_status_noalloc,
                     bakron_last_cuda_error, dequantize, factors_bytes, lib, library_path,
                     strerror, workspace_bytes)
from .buildlib import build  # noqa: F401
