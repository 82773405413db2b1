// The solve's internal entry point, shared by the C ABI (capi.cu), the
// no-allocation variant (noalloc.cu), the autotuner (tune.cu) and the batched
// solve (batch.cu).  Defined in solve.cu.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "tune.cuh"

namespace bakron {

// One BaKron solve of W (m x n) enqueued on `s` (arguments as bakron_solve,
// validated by the caller).  qmax: codes 0..qmax.  force: schedule to use
// instead of the per-shape table.  grid_given: scales/zeros hold the caller's
// grid (read only) instead of being computed.  keep_status: leave the
// workspace's status word as it is (a batch of solves keeps its first error).
int solve_impl(const void* W, int wdt, int m, int n, int64_t ldw, const void* factors, int qmax,
               int group_size, uint8_t* codes, float* scales, float* zeros, float* prerounding,
               void* workspace, cudaStream_t s, const Tuning* force, bool grid_given,
               bool keep_status);

// H <= 32 problems of one shape solved side by side, problem h in the
// workspace slice `slice` bytes after problem h - 1's: each tile anti-diagonal's
// leaves of all problems in one launch on `main`, each node's tensor-core band
// stages of all problems in one launch each on `main`, a narrower node's
// CUDA-core band products per problem on lanes[h]; the lanes must have been
// forked from `main` (an event recorded on main and waited on by every
// lane), and the caller joins them back afterwards; status words are cleared
// by the caller.  Returns
// BAKRON_ERR_INVALID_ARG, enqueueing nothing, when the shape's schedule uses
// dataflow leaves or persistent subtrees (the caller then runs the problems
// one by one on the lanes).
int solve_heads_impl(int H, const void* const* W, int wdt, int m, int n, int64_t ldw,
                     const void* const* factors, int qmax, int group_size,
                     uint8_t* const* codes, float* const* scales, float* const* zeros,
                     char* workspace, size_t slice, cudaStream_t main,
                     const cudaStream_t* lanes, cudaEvent_t fork, const cudaEvent_t* done);

// The B = I (GPTQ) solve (gptq.cu): grid, X from W, then the column
// recursion.  Workspace and factor buffer as the general solve (only L^A's
// planes and leaf blocks are read; the M planes hold E row-major).  Requires
// group_size == 0 or a multiple of 32 (a group covers whole tiles).
int gptq_impl(const void* W, int wdt, int m, int n, int64_t ldw, const void* factors, int qmax,
              int group_size, uint8_t* codes, float* scales, float* zeros, float* prerounding,
              void* workspace, cudaStream_t s);

// Diagnostic only (bakron_diag_leaf_chain): when set, the leaves of the next
// solve record the chain warp's clock64 before and after its 63 steps there.
extern long long* g_diag_leaf_clk;

}  // namespace bakron
