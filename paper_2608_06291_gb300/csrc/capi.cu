// C entry points of libbakron.so (declared in include/bakron.h): host-side
// validation, buffer sizes, factor import/export and the status word.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include <mutex>

#include "common.cuh"
#include "tune.cuh"
#include "solve.cuh"

namespace bakron {
int prepare_impl(const float* A, const float* B, int m, int n, float damp, void* factors,
                 void* workspace, cudaStream_t s);
int launch_grid_sym(const void* W, int wdt, int m, int n, int64_t ldw, int levels,
                    int group_size, int shrink_steps, float* scales, float* zeros,
                    cudaStream_t s);

// Largest side accepted.  Keeps every index product inside int64 and every
// grid dimension inside CUDA's limits (mp / 32 tiles per side).
constexpr int MAX_DIM = 1 << 17;

static bool dims_ok(int m, int n) { return m >= 1 && n >= 1 && m <= MAX_DIM && n <= MAX_DIM; }

// Dense unit-lower L (d x d, row-major, only the strictly-lower part read)
// into the padded factor section (Lp x Lp) with ones on the diagonal, zeros
// above it and an identity extension.
__global__ void k_import(const float* L, int d, float* hi, float* lo, int64_t Lp) {
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= Lp * Lp) return;
  const int64_t i = idx / Lp, j = idx % Lp;
  float v = (i == j) ? 1.f : 0.f;
  if (i < d && j < d && j < i) v = L[i * d + j];
  const float h = tf32_hi(v);
  hi[idx] = h;
  lo[idx] = v - h;
}

__global__ void k_import_diag(const float* r, int d, float* dst, int64_t Lp) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i < Lp) dst[i] = (r && i < d) ? r[i] : 1.f;
}

__global__ void k_export(const float* hi, const float* lo, int64_t Lp, int d, float* L) {
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= (int64_t)d * d) return;
  const int64_t k = (idx / d) * Lp + idx % d;
  L[idx] = hi[k] + lo[k];
}

static unsigned nblocks(int64_t work, int threads) { return (unsigned)((work + threads - 1) / threads); }

thread_local cudaError_t t_cuda_err = cudaSuccess;
thread_local const char* t_cuda_file = nullptr;
thread_local int t_cuda_line = 0;

int cuda_fail(cudaError_t e, const char* file, int line) {
  t_cuda_err = e;
  const char* base = file;
  for (const char* c = file; c && *c; ++c)
    if (*c == '/') base = c + 1;
  t_cuda_file = base;
  t_cuda_line = line;
  return BAKRON_ERR_CUDA;
}

}  // namespace bakron

using namespace bakron;

extern "C" {

size_t bakron_factors_bytes(int m, int n) {
  if (!dims_ok(m, n)) return 0;
  return FactorLayout(m, n).bytes;
}

size_t bakron_workspace_bytes(int m, int n) {
  if (!dims_ok(m, n)) return 0;
  size_t a = SolveLayout(m, n).bytes, b = PrepareLayout(m, n).bytes;
  return a > b ? a : b;
}

int bakron_prepare(const float* A, const float* B, int m, int n, float damp, void* factors,
                   void* workspace, size_t workspace_bytes, void* stream) {
  if (!A || !B || !factors || !workspace || !dims_ok(m, n) || !(damp >= 0.f))
    return BAKRON_ERR_INVALID_ARG;
  if (workspace_bytes < PrepareLayout(m, n).bytes) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  int rc = prepare_impl(A, B, m, n, damp, factors, workspace, s);
  if (rc != BAKRON_OK) return rc;
  return bakron_read_status(workspace, stream);
}

int bakron_set_factors(const float* LA, const float* LB, const float* rA, const float* rB, int m,
                       int n, void* factors, void* stream) {
  if (!LA || !LB || !factors || !dims_ok(m, n)) return BAKRON_ERR_INVALID_ARG;
  FactorLayout fl(m, n);
  cudaStream_t s = (cudaStream_t)stream;
  char* f = (char*)factors;
  k_import<<<nblocks(fl.np * fl.np, 256), 256, 0, s>>>(LA, n, (float*)(f + fl.off_LAH),
                                                       (float*)(f + fl.off_LAL), fl.np);
  k_import<<<nblocks(fl.mp * fl.mp, 256), 256, 0, s>>>(LB, m, (float*)(f + fl.off_LBH),
                                                       (float*)(f + fl.off_LBL), fl.mp);
  k_import_diag<<<nblocks(fl.np, 256), 256, 0, s>>>(rA, n, (float*)(f + fl.off_rA), fl.np);
  k_import_diag<<<nblocks(fl.mp, 256), 256, 0, s>>>(rB, m, (float*)(f + fl.off_rB), fl.mp);
  BK_CUDA_OK(cudaGetLastError());
  return build_leaf_blocks(fl, f, s);
}

int bakron_get_factors(const void* factors, int m, int n, float* LA, float* LB, float* rA,
                       float* rB, void* stream) {
  if (!factors || !dims_ok(m, n)) return BAKRON_ERR_INVALID_ARG;
  FactorLayout fl(m, n);
  cudaStream_t s = (cudaStream_t)stream;
  const char* f = (const char*)factors;
  if (LA)
    k_export<<<nblocks((int64_t)n * n, 256), 256, 0, s>>>(
        (const float*)(f + fl.off_LAH), (const float*)(f + fl.off_LAL), fl.np, n, LA);
  if (LB)
    k_export<<<nblocks((int64_t)m * m, 256), 256, 0, s>>>(
        (const float*)(f + fl.off_LBH), (const float*)(f + fl.off_LBL), fl.mp, m, LB);
  if (rA) BK_CUDA_OK(cudaMemcpyAsync(rA, f + fl.off_rA, sizeof(float) * n, cudaMemcpyDeviceToDevice, s));
  if (rB) BK_CUDA_OK(cudaMemcpyAsync(rB, f + fl.off_rB, sizeof(float) * m, cudaMemcpyDeviceToDevice, s));
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}

int bakron_solve(const void* W, int wdtype, int m, int n, int64_t ldw, const void* factors,
                 int bits, int group_size, uint8_t* codes, float* scales, float* zeros,
                 float* prerounding, void* workspace, size_t workspace_bytes, int sync,
                 void* stream) {
  if (!W || !factors || !codes || !scales || !zeros || !workspace || !dims_ok(m, n))
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || bits < 1 || bits > 8) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  if (workspace_bytes < SolveLayout(m, n).bytes) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  int rc = solve_impl(W, wdtype, m, n, ldw, factors, (1 << bits) - 1, group_size, codes, scales,
                      zeros, prerounding, workspace, s, nullptr, false, false);
  if (rc != BAKRON_OK || !sync) return rc;
  return bakron_read_status(workspace, stream);
}

int bakron_solve_gptq(const void* W, int wdtype, int m, int n, int64_t ldw, const void* factors,
                      int bits, int group_size, uint8_t* codes, float* scales, float* zeros,
                      float* prerounding, void* workspace, size_t workspace_bytes, int sync,
                      void* stream) {
  if (!W || !factors || !codes || !scales || !zeros || !workspace || !dims_ok(m, n))
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || bits < 1 || bits > 8) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && (n % group_size != 0 || group_size % TILE != 0)))
    return BAKRON_ERR_INVALID_ARG;
  if (workspace_bytes < SolveLayout(m, n).bytes) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  int rc = gptq_impl(W, wdtype, m, n, ldw, factors, (1 << bits) - 1, group_size, codes, scales,
                     zeros, prerounding, workspace, s);
  if (rc != BAKRON_OK || !sync) return rc;
  return bakron_read_status(workspace, stream);
}

int bakron_grid_symmetric(const void* W, int wdtype, int m, int n, int64_t ldw, int levels,
                          int group_size, int shrink_steps, float* scales, float* zeros,
                          void* stream) {
  if (!W || !scales || !zeros || !dims_ok(m, n)) return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || levels < 1 || levels > 127) return BAKRON_ERR_INVALID_ARG;
  if (shrink_steps < 0 || shrink_steps > 1024) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  return launch_grid_sym(W, wdtype, m, n, ldw, levels, group_size, shrink_steps, scales, zeros,
                         (cudaStream_t)stream);
}

int bakron_solve_with_grid(const void* W, int wdtype, int m, int n, int64_t ldw,
                           const void* factors, int qmax, int group_size, const float* scales,
                           const float* zeros, uint8_t* codes, float* prerounding,
                           void* workspace, size_t workspace_bytes, int sync, void* stream) {
  if (!W || !factors || !codes || !scales || !zeros || !workspace || !dims_ok(m, n))
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || qmax < 1 || qmax > 255) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  if (workspace_bytes < SolveLayout(m, n).bytes) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  // the grid is only read when grid_given is set
  int rc = solve_impl(W, wdtype, m, n, ldw, factors, qmax, group_size, codes,
                      const_cast<float*>(scales), const_cast<float*>(zeros), prerounding,
                      workspace, s, nullptr, true, false);
  if (rc != BAKRON_OK || !sync) return rc;
  return bakron_read_status(workspace, stream);
}

int bakron_read_status(void* workspace, void* stream) {
  if (!workspace) return BAKRON_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  int h = 0;
  BK_CUDA_OK(cudaMemcpyAsync(&h, workspace, sizeof(int), cudaMemcpyDeviceToHost, s));
  BK_CUDA_OK(cudaStreamSynchronize(s));
  BK_CUDA_OK(cudaMemsetAsync(workspace, 0, sizeof(int), s));
  BK_CUDA_OK(cudaGetLastError());
  return h;
}

int bakron_diag_leaf_chain(const void* W, int wdtype, const void* factors, uint8_t* codes,
                           float* scales, float* zeros, void* workspace, size_t workspace_bytes,
                           double* cycles_per_step, void* stream) {
  if (!W || !factors || !codes || !scales || !zeros || !workspace || !cycles_per_step)
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  const size_t need = SolveLayout(TILE, TILE).bytes;
  if (workspace_bytes < need + 256) return BAKRON_ERR_WORKSPACE;
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  cudaStream_t s = (cudaStream_t)stream;
  long long* clk = (long long*)((char*)workspace + need);
  BK_CUDA_OK(cudaMemsetAsync(clk, 0, 2 * sizeof(long long), s));
  g_diag_leaf_clk = clk;
  const int rc = solve_impl(W, wdtype, TILE, TILE, TILE, factors, 15, 0, codes, scales, zeros,
                            nullptr, workspace, s, nullptr, false, false);
  g_diag_leaf_clk = nullptr;
  if (rc != BAKRON_OK) return rc;
  long long h[2] = {0, 0};
  BK_CUDA_OK(cudaMemcpyAsync(h, clk, sizeof(h), cudaMemcpyDeviceToHost, s));
  BK_CUDA_OK(cudaStreamSynchronize(s));
  *cycles_per_step = (double)(h[1] - h[0]) / (2 * TILE - 1);
  return bakron_read_status(workspace, stream);
}

int bakron_last_cuda_error(const char** name, const char** where, int* line) {
  const int code = (int)t_cuda_err;
  if (name) *name = cudaGetErrorName(t_cuda_err);
  if (where) *where = t_cuda_file ? t_cuda_file : "";
  if (line) *line = t_cuda_line;
  return code;
}

const char* bakron_strerror(int status) {
  switch (status) {
    case BAKRON_OK: return "ok";
    case BAKRON_ERR_INVALID_ARG: return "invalid argument";
    case BAKRON_ERR_NOT_SPD: return "damped Gram is not positive definite";
    case BAKRON_ERR_CUDA: return "CUDA runtime error";
    case BAKRON_ERR_TIMEOUT: return "bounded device wait timed out";
    case BAKRON_ERR_WORKSPACE: return "workspace too small";
    case BAKRON_ERR_NONFINITE: return "non-finite value while rounding";
    default: return "unknown status";
  }
}

}  // extern "C"
