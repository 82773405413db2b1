"""CPU float64 oracle for the BaKron solver.

Test infrastructure only: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline legs of ``bench.py``, never by the product path.
"""
from .bakron_oracle import *  # noqa: F401,F403
from .bakron_oracle import (Factors, Grid, Result, bakron, bakron_antidiagonal,  # noqa: F401
                            bakron_naive, bakron_recursive, bakron_vectorized,
                            brute_force, certificate, damped, dequantize,
                            error_bound, gptq_rows, integer_grid, midpoint_distance,
                            objective, objective_from_errors, prepare, quant_grid,
                            quantize, rev_cholesky, rtn, teacher_forced,
                            unit_lower_factor, unit_lower_factor_via_rev,
                            certificate_rows, grid_rows)
from .hessian import (gram, kfac_factors, kronecker_hessian, rearranged_hessian,  # noqa: F401
                      sample_quadforms, sample_sqnorms, shampoo_factors)
