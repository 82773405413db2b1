// Measured issue rate of the tensor-core instruction the band products use
// (tcgen05.mma kind::tf32, M = 128, N = 128, K = 8, one CTA per SM), for the
// tensor roofline of the solve: bakron_diag_mma_rate (include/bakron.h).
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "tc_gemm.cuh"

namespace bakron {
namespace {

constexpr int RM = 128, RN = 128, RK = 32;   // one 32-deep K stage of operands in shared memory

__device__ __forceinline__ uint32_t s_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// K-major operand, 128-byte swizzle, 8-row groups 1024 bytes apart, version 1.
__device__ __forceinline__ uint64_t s_desc(uint32_t addr) {
  return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Each CTA issues `stages` x 4 MMAs (K = 8 each) into one TMEM accumulator
// from operands resident in shared memory (no loads), then waits, for at
// most `limit` cycles, for them to complete.  Writes its elapsed cycles.
__global__ void __launch_bounds__(128, 1)
k_mma_rate(int stages, long long limit, long long* cycles, int* status) {
  extern __shared__ __align__(1024) unsigned char raw[];
  unsigned char* sm = (unsigned char*)(((uintptr_t)raw + 1023) & ~(uintptr_t)1023);
  __shared__ uint64_t bar;
  __shared__ uint32_t tslot;
  const int t = threadIdx.x, warp = t >> 5;
  for (int i = t; i < (RM + RN) * RK; i += blockDim.x) {
    const unsigned h = (unsigned)i * 2654435761u + 12345u;
    ((float*)sm)[i] = (float)(h >> 8) * (1.0f / 16777216.f) - 0.5f;
  }
  if (t == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(s_u32(&bar)), "r"(1));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     s_u32(&tslot)),
                 "r"(RN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tslot;
  if (t == 0) {
    const uint64_t da = s_desc(s_u32(sm)), db = s_desc(s_u32(sm) + RM * RK * 4);
    const uint32_t idesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(RN >> 3) << 17) |
                           ((uint32_t)(RM >> 4) << 24);
    const long long t0 = clock64();
    for (int i = 0; i < stages; ++i) {
#pragma unroll
      for (int kk = 0; kk < RK / 8; ++kk) {
        const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
        asm volatile(
            "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
            "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem),
            "l"(da + 2 * kk), "l"(db + 2 * kk), "r"(idesc), "r"(acc)
            : "memory");
      }
    }
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            s_u32(&bar))
        : "memory");
    uint32_t done = 0;
    const long long w0 = clock64();
    while (!done) {
      asm volatile(
          "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
          "selp.u32 %0, 1, 0, p;\n\t}"
          : "=r"(done)
          : "r"(s_u32(&bar)), "r"(0)
          : "memory");
      if (!done && clock64() - w0 > limit) {
        atomicCAS(status, 0, BAKRON_ERR_TIMEOUT);
        break;
      }
    }
    cycles[blockIdx.x] = clock64() - t0;
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(RN)
                 : "memory");
}

}  // namespace
}  // namespace bakron

using namespace bakron;

extern "C" int bakron_diag_mma_rate(int stages, void* workspace, size_t workspace_bytes,
                                    double* tflops, double* cycles_per_mma, void* stream) {
  if (stages < 1 || stages > (1 << 20) || !workspace || !tflops) return BAKRON_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  BK_CUDA_OK(cudaGetDevice(&dev));
  BK_CUDA_OK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  if (workspace_bytes < 256 + sizeof(long long) * (size_t)sms) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  int* status = (int*)ws;
  long long* cyc = (long long*)(ws + 256);
  const int smem = (RM + RN) * RK * 4 + 1024;
  BK_CUDA_OK(cudaFuncSetAttribute(k_mma_rate, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  BK_CUDA_OK(cudaMemsetAsync(status, 0, 256, s));
  const long long limit = spin_cycles_from_env();
  k_mma_rate<<<sms, 128, smem, s>>>(stages, limit, cyc, status);   // warm-up
  cudaEvent_t e0, e1;
  BK_CUDA_OK(cudaEventCreate(&e0));
  if (cudaEventCreate(&e1) != cudaSuccess) {
    cudaEventDestroy(e0);
    return BAKRON_ERR_CUDA;
  }
  cudaEventRecord(e0, s);
  k_mma_rate<<<sms, 128, smem, s>>>(stages, limit, cyc, status);
  cudaEventRecord(e1, s);
  int rc = BAKRON_OK;
  float ms = 0.f;
  if (cudaEventSynchronize(e1) != cudaSuccess || cudaEventElapsedTime(&ms, e0, e1) != cudaSuccess)
    rc = BAKRON_ERR_CUDA;
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (rc != BAKRON_OK) return rc;
  long long c0 = 0;
  BK_CUDA_OK(cudaMemcpy(&c0, cyc, sizeof(c0), cudaMemcpyDeviceToHost));
  const int st = bakron_read_status(workspace, stream);
  if (st != BAKRON_OK) return st;
  const double mmas = 4.0 * stages;
  *tflops = 2.0 * RM * RN * 8 * mmas * sms / (ms * 1e-3) / 1e12;
  if (cycles_per_mma) *cycles_per_mma = (double)c0 / mmas;
  return BAKRON_OK;
}
