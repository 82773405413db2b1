// bakron_solve_noalloc: the solve for callers that cannot allocate device
// memory.  Its scratch is a fixed array in this file instead of a caller
// workspace; everything else is bakron_solve.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "tune.cuh"
#include "solve.cuh"

namespace bakron {

// The scratch.  Every GPU that loads the library holds it until the process
// exits.  In host code this name is only a stand-in for the device symbol:
// its device address comes from cudaGetSymbolAddress, once per context.
static __device__ __align__(256) unsigned char g_noalloc_scratch[BAKRON_NOALLOC_SCRATCH_BYTES];

namespace {
std::mutex g_noalloc_mu;
// context id -> scratch address.  Keyed on the context rather than the device
// ordinal: after a device reset (or the primary context being destroyed and
// made again) the module is loaded anew and the array may live elsewhere;
// the new context has a new id, so its address is looked up again.
std::unordered_map<unsigned long long, void*> g_noalloc_addr;

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);
CtxGetCurrentFn g_ctx_current = nullptr;
CtxGetIdFn g_ctx_id = nullptr;

// The driver calls that name the current context, taken through the runtime
// (the library links no driver library).  Caller holds g_noalloc_mu.
cudaError_t driver_calls() {
  if (g_ctx_current && g_ctx_id) return cudaSuccess;
  cudaDriverEntryPointQueryResult q1, q2;
  void *f1 = nullptr, *f2 = nullptr;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f1, 12000,
                                                   cudaEnableDefault, &q1);
  if (e != cudaSuccess || q1 != cudaDriverEntryPointSuccess || !f1) return cudaErrorNotSupported;
  e = cudaGetDriverEntryPointByVersion("cuCtxGetId", &f2, 12000, cudaEnableDefault, &q2);
  if (e != cudaSuccess || q2 != cudaDriverEntryPointSuccess || !f2) return cudaErrorNotSupported;
  g_ctx_current = (CtxGetCurrentFn)f1;
  g_ctx_id = (CtxGetIdFn)f2;
  return cudaSuccess;
}

// Id of the current context, 0 if none is current yet.
cudaError_t current_ctx_id(unsigned long long* id) {
  CUcontext c = nullptr;
  *id = 0;
  if (g_ctx_current(&c) != CUDA_SUCCESS) return cudaErrorUnknown;
  if (!c) return cudaSuccess;
  return g_ctx_id(c, id) == CUDA_SUCCESS ? cudaSuccess : cudaErrorUnknown;
}

// Device address of the scratch in the current context (looked up on the
// first use in that context).
cudaError_t noalloc_scratch(void** out) {
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  cudaError_t e = driver_calls();
  if (e != cudaSuccess) return e;
  unsigned long long id = 0;
  if ((e = current_ctx_id(&id)) != cudaSuccess) return e;
  if (id != 0) {
    auto it = g_noalloc_addr.find(id);
    if (it != g_noalloc_addr.end()) {
      *out = it->second;
      return cudaSuccess;
    }
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_noalloc_scratch);   // makes the device's context current
  if (e != cudaSuccess) return e;
  if (id == 0 && (e = current_ctx_id(&id)) != cudaSuccess) return e;
  if (id != 0) g_noalloc_addr[id] = p;
  *out = p;
  return cudaSuccess;
}

constexpr int MAX_SIDE = 1 << 17;   // as bakron_solve
}  // namespace
}  // namespace bakron

extern "C" int bakron_solve_noalloc(const void* W, int wdtype, int m, int n, int64_t ldw,
                                    const void* factors, int bits, int group_size,
                                    uint8_t* codes, float* scales, float* zeros,
                                    float* prerounding, int sync, void* stream) {
  using namespace bakron;
  if (!W || !factors || !codes || !scales || !zeros || m < 1 || n < 1)
    return BAKRON_ERR_INVALID_ARG;
  if (m > MAX_SIDE || n > MAX_SIDE) return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || bits < 1 || bits > 8) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  if (SolveLayout(m, n).bytes > BAKRON_NOALLOC_SCRATCH_BYTES) return BAKRON_ERR_WORKSPACE;
  void* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) return BAKRON_ERR_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  int rc = solve_impl(W, wdtype, m, n, ldw, factors, (1 << bits) - 1, group_size, codes, scales,
                      zeros, prerounding, scratch, s, nullptr, false, false);
  if (rc != BAKRON_OK || !sync) return rc;
  return bakron_read_status(scratch, stream);
}

extern "C" int bakron_read_status_noalloc(void* stream) {
  using namespace bakron;
  void* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) return BAKRON_ERR_CUDA;
  return bakron_read_status(scratch, stream);
}
