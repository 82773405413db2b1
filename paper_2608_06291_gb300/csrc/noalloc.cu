// bakron_solve_noalloc: the solve for callers that cannot allocate device
// memory.  Its scratch is a fixed array in this file instead of a caller
// workspace; everything else is bakron_solve.
#include <cuda_runtime.h>

#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "tune.cuh"
#include "solve.cuh"

namespace bakron {

// The scratch.  Every GPU that loads the library holds it until the process
// exits.  In host code this name is only a stand-in for the device symbol:
// its device address comes from cudaGetSymbolAddress, once per device.
static __device__ __align__(256) unsigned char g_noalloc_scratch[BAKRON_NOALLOC_SCRATCH_BYTES];

namespace {
std::mutex g_noalloc_mu;
std::unordered_map<int, void*> g_noalloc_addr;   // device ordinal -> scratch address

// Device address of the scratch on the current device (set up on first use).
cudaError_t noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  auto it = g_noalloc_addr.find(dev);
  if (it != g_noalloc_addr.end()) {
    *out = it->second;
    return cudaSuccess;
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return e;
  g_noalloc_addr[dev] = p;
  *out = p;
  return cudaSuccess;
}
}  // namespace
}  // namespace bakron

extern "C" int bakron_solve_noalloc(const void* W, int wdtype, int m, int n, int64_t ldw,
                                    const void* factors, int bits, int group_size,
                                    uint8_t* codes, float* scales, float* zeros,
                                    float* prerounding, int sync, void* stream) {
  using namespace bakron;
  if (!W || !factors || !codes || !scales || !zeros || m < 1 || n < 1)
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || bits < 1 || bits > 8) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  if (m > (1 << 17) || n > (1 << 17)) return BAKRON_ERR_WORKSPACE;
  if (SolveLayout(m, n).bytes > BAKRON_NOALLOC_SCRATCH_BYTES) return BAKRON_ERR_WORKSPACE;
  void* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) return BAKRON_ERR_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  int rc = solve_impl(W, wdtype, m, n, ldw, factors, (1 << bits) - 1, group_size, codes, scales,
                      zeros, prerounding, scratch, s, nullptr, false, false);
  if (rc != BAKRON_OK || !sync) return rc;
  return bakron_read_status(scratch, stream);
}
