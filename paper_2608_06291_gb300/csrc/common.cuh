// Shared definitions of the BaKron CUDA library: buffer layouts, tile sizes,
// status handling.  Everything here is internal; the C ABI is include/bakron.h.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/bakron.h"

namespace bakron {

// Leaf tile: one warp rounds a TILE x TILE block of W by walking its
// 2*TILE-1 anti-diagonals (lane = column).
constexpr int TILE = 32;
// All matrices are padded to this multiple in both dimensions, so that the
// GEMM kernels see whole 128 x 128 blocks and TMA boxes never straddle an edge.
constexpr int PAD = 128;

__host__ __device__ inline int64_t round_up(int64_t x, int64_t r) {
  return (x + r - 1) / r * r;
}
__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Split of an fp32 value into an exact tf32 head and an fp32 tail:
// hi = x rounded to the nearest value with 10 mantissa bits (the 13 low bits
// cleared after adding half of their range), lo = x - hi, exact in fp32 with
// |lo| <= 2^-11 |x|, so hi + lo == x exactly.  Rounding (not truncating) hi
// makes lo symmetric around zero, so the tensor core's truncation of lo to
// tf32 errs with random sign instead of always toward x: no bias builds up
// over long contractions.
__host__ __device__ inline float tf32_hi(float x) {
#ifdef __CUDA_ARCH__
  return __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xFFFFE000u);
#else
  union { float f; uint32_t u; } v;
  v.f = x;
  v.u = (v.u + 0x1000u) & 0xFFFFE000u;
  return v.f;
#endif
}

// Factor buffer: [L^B hi][L^B lo] (mp x mp each) [L^A hi][L^A lo] (np x np)
// [rB mp][rA np], fp32, sections 256-byte aligned.  L^X = hi + lo exactly;
// stored dense row-major with exact zeros above the diagonal, ones on it and
// an identity extension over the padding.
// Then the leaf blocks: per tile row I of L^B, the diagonal block and the
// LEAF_BLOCKS - 1 blocks left of it, L^B[I, I - d]; per tile column J of L^A,
// L^A[J, J - g]; fp32 (hi + lo), TILE rows of LEAF_BLOCK_LD floats each (the
// columns past TILE zero), laid out as the leaf kernel keeps them in shared
// memory (see build_leaf_blocks), so that it copies them as they are.
constexpr int LEAF_BLOCKS = 16;
constexpr int LEAF_BLOCK_LD = 36;
constexpr int LEAF_BLOCK_FLOATS = TILE * LEAF_BLOCK_LD;

struct FactorLayout {
  int m, n;
  int64_t mp, np, Mt, Nt;
  size_t off_LBH, off_LBL, off_LAH, off_LAL, off_rB, off_rA, off_LBblk, off_LAblk, bytes;
  explicit FactorLayout(int m_, int n_) : m(m_), n(n_) {
    mp = round_up(m, PAD);
    np = round_up(n, PAD);
    Mt = mp / TILE;
    Nt = np / TILE;
    off_LBH = 0;
    off_LBL = align256(off_LBH + size_t(mp * mp) * 4);
    off_LAH = align256(off_LBL + size_t(mp * mp) * 4);
    off_LAL = align256(off_LAH + size_t(np * np) * 4);
    off_rB = align256(off_LAL + size_t(np * np) * 4);
    off_rA = align256(off_rB + size_t(mp) * 4);
    off_LBblk = align256(off_rA + size_t(np) * 4);
    off_LAblk = align256(off_LBblk + size_t(Mt) * LEAF_BLOCKS * LEAF_BLOCK_FLOATS * 4);
    bytes = align256(off_LAblk + size_t(Nt) * LEAF_BLOCKS * LEAF_BLOCK_FLOATS * 4);
  }
};

// Fills the leaf blocks of a factor buffer from its L^B and L^A planes
// (solve.cu); run after every write of the planes.
int build_leaf_blocks(const FactorLayout& fl, char* factors, cudaStream_t s);

// Solve workspace: [status 256 B][X mp x np][E^T hi, lo: np x mp each]
// [M hi, lo: mp x np each], fp32.  X holds W widened and, once an entry is
// rounded, the value it was rounded at.  E^T is the error matrix transposed
// (row = column index of W) so that it is K-major as the second operand of
// M = L^B E; M is the stage-1 band product.  The M hi plane doubles as E^T in
// fp32 for the leaves: a leaf block reads back only E tiles written inside the
// block, and M is written only by band products, which run between blocks.
// Then the leaves' dataflow words (one launch per block of leaves): a tile
// counter per block, indexed by the block's first anti-diagonal, and a
// readiness flag per padded tile; zeroed at the start of every solve.
constexpr int FLOW_COUNTERS = 8192;   // > the anti-diagonals of the largest problem (2 * 4096)
struct SolveLayout {
  int64_t mp, np;
  size_t off_status, off_X, off_EtH, off_EtL, off_MH, off_ML, off_flow, flow_bytes, bytes;
  SolveLayout(int m, int n) {
    mp = round_up(m, PAD);
    np = round_up(n, PAD);
    const size_t plane = size_t(mp * np) * 4;
    off_status = 0;
    off_X = 256;
    off_EtH = align256(off_X + plane);
    off_EtL = align256(off_EtH + plane);
    off_MH = align256(off_EtL + plane);
    off_ML = align256(off_MH + plane);
    off_flow = align256(off_ML + plane);
    flow_bytes = size_t(FLOW_COUNTERS + (mp / TILE) * (np / TILE)) * 4;
    bytes = align256(off_flow + flow_bytes);
  }
};

// Prepare works on one Gram at a time (the larger side bounds the size).
// Real type of the factorisation: fp64 (see prepare.cu for the reason).
struct PrepareLayout {
  int64_t dp;
  size_t off_status, off_C, off_Linv, off_T, off_scalar, bytes;
  PrepareLayout(int m, int n) {
    int64_t d = m > n ? m : n;
    dp = round_up(d, PAD);
    off_status = 0;
    off_C = 256;
    off_Linv = align256(off_C + size_t(dp * dp) * 8);
    off_T = align256(off_Linv + size_t(dp * dp) * 8);
    off_scalar = align256(off_T + size_t(dp * PAD) * 8);
    bytes = align256(off_scalar + 256);
  }
};

// Programmatic dependent launch.  Every kernel of the solve waits for the
// previous kernel on the stream to complete (pdl_wait) before it touches data
// that kernel or its predecessors wrote, and only then lets the next kernel
// launch (pdl_trigger).  So the next kernel's launch and prologue overlap this
// kernel's work, and anything it reads before its own pdl_wait was produced at
// least two kernels earlier.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Timeline stamps of one kernel launch (benchmark instrumentation; kernels
// receive a null slot unless bakron_profile_enable(2) is on): slot[0] takes
// the earliest time a CTA of the launch started its dependent work (after its
// pdl_wait), slot[1] the latest time a CTA finished, in %globaltimer
// nanoseconds.  Thread 0 of each CTA stamps.
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void stamp_begin(unsigned long long* slot) {
  if (slot != nullptr && threadIdx.x == 0) atomicMin(slot, global_ns());
}
__device__ __forceinline__ void stamp_end(unsigned long long* slot) {
  if (slot != nullptr && threadIdx.x == 0) atomicMax(slot + 1, global_ns());
}

// tf32 split of an fp32 value: hi = x rounded to tf32, lo = the rest rounded
// to tf32 (the 3xTF32 scheme: products hi*hi + hi*lo + lo*hi keep fp32
// accuracy; the dropped lo*lo term is below 2^-22 relative).
__device__ __forceinline__ void tf32_split(float x, uint32_t& hi, uint32_t& lo) {
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(hi) : "f"(x));
  const float rest = x - __uint_as_float(hi);
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(lo) : "f"(rest));
}

// D += A B on the warp's tensor cores (mma.sync; used for the small 32^3
// products of the leaves): A 16 x 8 (row-major fragment a[4]),
// B 8 x 8 (b[2]), D 16 x 8 fp32 (d[4]), tf32 inputs.
__device__ __forceinline__ void mma_tf32_16x8x8(float (&d)[4], const uint32_t (&a)[4],
                                                const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// Device status word (first int of every workspace).  Kernels only ever raise
// it with atomicMax-free writes of a nonzero code; the host reads and clears.
__device__ inline void raise_status(int* status, int code) {
  atomicCAS(status, 0, code);
}

}  // namespace bakron

namespace bakron {
// Records, for the calling host thread, the CUDA runtime error behind a
// BAKRON_ERR_CUDA and where the library saw it (bakron_last_cuda_error);
// returns BAKRON_ERR_CUDA.
int cuda_fail(cudaError_t e, const char* file, int line);
}  // namespace bakron

#define BK_CUDA_OK(expr)                                                      \
  do {                                                                        \
    cudaError_t err__ = (expr);                                               \
    if (err__ != cudaSuccess) return ::bakron::cuda_fail(err__, __FILE__, __LINE__); \
  } while (0)

// BAKRON_OK, or BAKRON_ERR_CUDA with the error recorded.
#define BK_CUDA_RC(expr)                                                      \
  ([&]() -> int {                                                             \
    cudaError_t err__ = (expr);                                               \
    return err__ == cudaSuccess ? BAKRON_OK : ::bakron::cuda_fail(err__, __FILE__, __LINE__); \
  }())
