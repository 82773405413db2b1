// Band products of Alg. 5 on the 5th-generation tensor cores (tcgen05), with
// FP32-accurate "3xTF32" arithmetic.
//
// The update between the two halves of an Alg. 5 node is two restricted band
// products (Appendix, complexity of BaKron):
//     stage 1:  M = L^B E_{S1}                 (E masked to the band S1)
//     stage 2:  X[S2] += Pi_{S2}(M L^A^T)      (only tiles of the band S2 written)
// Both are plain C = A B^T contractions with A and B K-major (row-major with
// the contraction index contiguous): stage 1 reads L^B (rows i, K = i') and
// E^T (rows j', K = i'); stage 2 reads M (rows i, K = j') and L^A (rows j,
// K = j').  Zeros of the triangular factors above their diagonal come from the
// data; the only masking is (a) stage-1 E sub-tiles outside S1, which are
// zero-filled in shared memory instead of loaded, and (b) stage-2 output
// tiles outside S2, which the epilogue leaves untouched.
//
// Precision: every operand is kept in global memory as a pair x = hi + lo
// (hi = x rounded to tf32, lo = x - hi exact in fp32), and
//     A B^T ~= A_hi B_hi^T + A_hi B_lo^T + A_lo B_hi^T,
// three kind::tf32 MMAs into one fp32 TMEM accumulator (the error-compensated
// split of Markidis et al. 2018 / Ootomo & Yokota 2022).  The dropped lo*lo
// term is <= 2^-22 relative and the tensor core's truncation of lo <= 2^-21,
// with random sign because hi is rounded to nearest.
//
// CTA (320 threads): warp 0 produces (TMA loads, zero fills), warp 1
// allocates TMEM and issues the MMAs (one thread), warps 2..9 sum the K
// stages: each 32-wide stage is accumulated afresh in one of four TMEM
// accumulators and added, in fp32 round-to-nearest, into registers by the two
// warps that own its 32-lane quarter (64 columns each, tcgen05.ld), while the
// MMAs of the next stages run.  The finished block goes out through shared
// memory (the freed ring, in the tensor maps' 128-byte swizzled layout) by
// TMA: stage 1 stores M as hi/lo planes, stage 2 adds into X with a TMA
// reduction, one 32 x 32 tile of S2 at a time.  One 128 x 128 output block per CTA, K staged
// 32 at a time through a 3-deep shared-memory ring.  The grid covers exactly
// the bounding box of the output blocks that have work (rows from row0).
// Every wait is bounded: a timed-out wait records BAKRON_ERR_TIMEOUT and the
// CTA winds down, draining its own TMA copies and MMAs (with a separate,
// generous limit) before it frees TMEM.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdint.h>
#include <stdlib.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "profile.cuh"
#include "tc_gemm.cuh"

namespace bakron {

namespace {

constexpr int BM = 128, BN = 128, BK = 32;     // output block and K stage (fp32 elements)
constexpr int STAGES = 3;
constexpr int EPI_WARPS = 8;                   // two per TMEM lane quarter
constexpr int THREADS = 32 * (2 + EPI_WARPS);
constexpr int EPI_COLS = BN / 2;               // columns summed by one epilogue warp
constexpr uint32_t TILE_BYTES = BM * BK * 4;   // 16 KiB: one operand plane of one stage
constexpr uint32_t STAGE_BYTES = 4 * TILE_BYTES;  // A hi, A lo, B hi, B lo
constexpr uint32_t SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;
constexpr int NACC = 4;                         // TMEM accumulators, rotating per K stage
constexpr uint32_t TMEM_COLS = NACC * BN;       // all 512 columns: one CTA per SM (shared memory)

// Paired variant (V_PAIR): two CTAs of a cluster compute the 128 x 128 blocks
// of two adjacent row blocks at the same column block with one M = 256
// MMA (cta_group::2).  Each CTA holds its own 128 rows of A and one half (64
// rows) of the shared B; the tensor cores of both SMs read both halves.  Per
// SM and 32-deep K stage that is 48 KiB written into shared memory by TMA and
// 72 KiB read by the MMAs, against 64 + 96 KiB for one CTA alone: shared
// memory bandwidth (about 128 B per cycle), not the tensor pipe, bounds the
// single-CTA kernel.  Four ring slots of 48 KiB.  Measured on GB300 it is
// slower than one CTA per block (4096^2 band stages 3.07 against 2.12 ms per
// solve, 28672 x 8192: 101 against 67 ms; the same with CTA-scope waits), so
// it is off by default (BAKRON_TC_PAIR=1 selects it).
constexpr int PAIR_STAGES = 4;
constexpr int BN_HALF = BN / 2;
constexpr uint32_t PAIR_STAGE_BYTES = 2 * TILE_BYTES + 2 * (TILE_BYTES / 2);
constexpr uint32_t PAIR_SMEM_BYTES = PAIR_STAGES * PAIR_STAGE_BYTES + 1024 + 256;
static_assert(PAIR_STAGES <= NACC, "a slot is freed by the commit of its accumulator");
static_assert(PAIR_STAGES * PAIR_STAGE_BYTES >= 8 * TILE_BYTES, "the epilogue stages 8 boxes in the ring");

// MODE_COLS: the column-band update of the B = I (GPTQ) schedule,
// X[:, S2] += E[:, S1] L^A[S2, S1]^T with S1 = tile columns [k, h) and S2 =
// [h, l); it reads and writes like stage 2 (A = E in the M planes, B = L^A,
// TMA reduce-add into X).
enum Mode { MODE_DENSE = 0, MODE_STAGE1 = 1, MODE_STAGE2 = 2, MODE_GRAM = 3, MODE_COLS = 4 };

struct TcParams {
  int mode;
  int k, h, l;          // band node (tile anti-diagonals), stage 1/2
  int Mt, Nt;           // real 32-tiles per side
  int row0;             // first output 128-block row (grid.y counts from here)
  int K;                // dense mode: contraction length (multiple of 32)
  float* out_hi;        // stage 1: M hi; dense: C
  float* out_lo;        // stage 1: M lo
  float* X;             // stage 2: accumulated in place
  int64_t ldo;          // leading dimension of out_hi/out_lo/X (elements)
  int* status;
  long long spin_cycles;  // bound of the working waits (clock64 cycles)
  // Gram mode: G <- beta G + alpha A B^T on the lower-triangle blocks, each
  // entry (i, j <= i) < dreal written and mirrored to (j, i); a_exact /
  // b_exact: that operand's lo plane is zero (skip its correction MMA)
  float alpha, beta;
  int dreal;
  int a_exact, b_exact;
  unsigned long long* stamp;   // timeline stamp slot of the launch (null: none)
  int raster;                  // band stages: row blocks per launch-order group (>= 1)
};

// Kernel variants (compile time, so that the band products' issue loop
// carries no Gram logic):
//   V_BAND      band products and the dense diagnostic: 3xTF32, one K stage
//               per TMEM accumulator, a slot freed by its accumulator's commit
//   V_GRAM_TF32 Gram on tf32 hi/lo planes; a_exact / b_exact skip the MMAs
//               of an operand whose lo plane is zero
//   V_GRAM_BF16 Gram on bf16 planes: mapA2 / mapB2 are plain bf16 maps (64 x
//               128 boxes), a ring slot holds one box of each (K = 64), the
//               MMAs are kind::f16 (bf16 x bf16 products exact in fp32), and
//               GRAM_KGROUP slots are summed in place per accumulator, each
//               slot freed by its own commit to `empty`
//   V_PAIR      band products and the dense diagnostic on CTA pairs (above)
enum Variant { V_BAND = 0, V_GRAM_TF32 = 1, V_GRAM_BF16 = 2, V_PAIR = 3 };

template <int V>
struct Ring {
  static constexpr bool pair = V == V_PAIR;
  static constexpr int stages = pair ? PAIR_STAGES : STAGES;
  static constexpr uint32_t b_plane = pair ? TILE_BYTES / 2 : TILE_BYTES;   // one B plane
  static constexpr uint32_t stage_bytes = 2 * TILE_BYTES + 2 * b_plane;
};
constexpr int GRAM_KGROUP = 4;
// Band products: K stages summed in place per TMEM accumulator (each group
// restarts its accumulator; the epilogue adds the groups in fp32).  Two
// stages per accumulator measured 1% faster per solve on GB300 but moved the
// 4096^2 free-running objective from 8e-5 to 3e-4 of the fp64 solve's (an
// earlier tie, then its cascade): one stage it is.
constexpr int BAND_KGROUP = 1;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// Adds to the bytes the current phase waits for, without arriving.
__device__ __forceinline__ void mbar_expect_tx_only(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `bar` with the given parity to complete, for at most
// `limit` cycles.  Returns false on time-out.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, long long limit) {
  if (mbar_test(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_test(bar, parity)) return true;
    if (clock64() - t0 > limit) return false;
  }
}

// A hi/lo plane pair in one copy: a rank-3 box (32 columns, rows, 2 planes)
// lands as the two planes one after the other (16 KiB each for 128 rows),
// each in the 128-byte swizzled layout; one box instead of two halves the
// TMA unit's per-box cost, which bounds the ring (measured on GB300: a 64 KiB
// slot of four 16 KiB boxes takes 0.62 us, of two 32 KiB boxes 0.45 us).
__device__ __forceinline__ void tma_load_pair(void* dst, const CUtensorMap* map, uint64_t* bar,
                                              int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(0)
      : "memory");
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row core groups 1024 bytes apart (SBO), version 1.
// TMA store of a box from shared memory, and TMA reduce-add of a box into
// global memory (fp32 add at L2), both tracked as a bulk group of the thread.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(smem_u32(src))
               : "memory");
}
__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* map, const void* src, int x, int y) {
  asm volatile(
      "cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(x), "r"(y), "r"(smem_u32(src))
      : "memory");
}
__device__ __forceinline__ void bulk_commit_and_wait() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFF) >> 4);            // start address
  d |= (uint64_t)1 << 16;                             // leading byte offset (unused, 1)
  d |= (uint64_t)(1024 >> 4) << 32;                   // stride byte offset
  d |= (uint64_t)1 << 46;                             // descriptor version
  d |= (uint64_t)2 << 61;                             // swizzle: 128 B
  return d;
}

// Instruction descriptor: kind::tf32, D fp32, A and B tf32 K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
  return (1u << 4)            // D format fp32
         | (2u << 7)          // A format tf32
         | (2u << 10)         // B format tf32
         | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_tf32(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Instruction descriptor: kind::f16 with bf16 A and B (K-major), D fp32, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4)            // D format fp32
         | (1u << 7)          // A format bf16
         | (1u << 10)         // B format bf16
         | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// ---- CTA-pair forms (cluster of two along y; rank 0 issues the MMAs)
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Address, in the cluster's shared window, of the same variable in rank 0.
__device__ __forceinline__ uint32_t at_rank0(const void* p) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(r) : "r"(smem_u32(p)));
  return r;
}

__device__ __forceinline__ void cmbar_arrive_expect_tx(uint32_t cbar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cluster.shared::cluster.b64 _, [%0], %1;" ::"r"(
                   cbar),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void cmbar_expect_tx_only(uint32_t cbar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cluster.shared::cluster.b64 [%0], %1;" ::"r"(cbar),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void cmbar_arrive(uint32_t cbar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cbar)
               : "memory");
}

// Bounded wait with cluster-scope acquire (arrivals from the other CTA).
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, long long limit) {
  const long long t0 = clock64();
  while (true) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
    if (clock64() - t0 > limit) return false;
  }
}

// TMA loads into this CTA's shared memory whose completion is counted on an
// mbarrier of rank 0 (cta_group::2: the barrier may sit in the peer CTA).
__device__ __forceinline__ void tma_load_pair_c2(void* dst, const CUtensorMap* map, uint32_t cbar,
                                                 int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(cbar), "r"(x), "r"(y), "r"(0)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d_c2(void* dst, const CUtensorMap* map, uint32_t cbar,
                                               int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(cbar), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void mma_tf32_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives on the barrier at this offset in both CTAs of the pair once every
// MMA issued so far has completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"((unsigned short)3)
      : "memory");
}

// Sets the int at this offset in the other CTA of the pair.
__device__ __forceinline__ void st_peer_flag(const void* local, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank ^ 1));
  asm volatile("st.relaxed.cluster.shared::cluster.u32 [%0], %1;" ::"r"(r), "r"(1u) : "memory");
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

// 32 lanes x 32 consecutive fp32 columns of TMEM into v (one per column) of
// each thread; the values are valid only after tmem_wait_ld().
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Output block and K range of this CTA.
struct Block {
  int rb, cb;         // output block (128-row block, 128-col block)
  int k0, nk;         // first K tile (32 wide) and number of K tiles the MMAs run
  int ok0, onk;       // the K tiles this block's own rows need (pairs: a subrange)
  bool own;           // the block is written (pairs: this CTA's row block has work)
};

// Column blocks [cb_lo, cb_hi] of 128-row block rb that have work in a band
// stage; false if the row block has none.  Shared by the kernel (which block
// is this CTA) and the host (the grid's bounding box).
__host__ __device__ inline bool band_row_span(int mode, int k, int h, int l, int Mt, int Nt, int rb,
                                              int& cb_lo, int& cb_hi) {
  const int I0 = 4 * rb;                     // first 32-tile row of the block
  if (I0 >= Mt) return false;
  if (mode == MODE_COLS) {                   // every row; output tile columns [h, l)
    cb_lo = h / 4;
    cb_hi = (l - 1) / 4;
    return true;
  }
  // output 32-tiles (I, J) of the band S2 = [h, l) in rows I0..I0+3
  const int Ilast = min(I0 + 3, Mt - 1);
  const int jout_lo = max(0, h - Ilast);
  const int jout_hi = min(Nt - 1, l - 1 - I0);
  if (jout_lo > jout_hi) return false;
  if (mode == MODE_STAGE1) {
    // M tiles (I, J') needed by stage 2 for these rows
    const int jp_lo = max(0, k - Ilast);
    const int jp_hi = min(h - 1, jout_hi);
    if (jp_lo > jp_hi) return false;
    cb_lo = jp_lo / 4;
    cb_hi = jp_hi / 4;
    return true;
  }
  cb_lo = jout_lo / 4;
  cb_hi = jout_hi / 4;
  return true;
}

// CTAs run in launch order, so consecutive ones should share operands in L2:
// the band stages walk their grid in groups of RASTER_ROWS row blocks, column
// by column inside a group (an A row block is then reused by the ~150
// resident CTAs of its group, and a B column block by RASTER_ROWS of them,
// instead of every B block coming from DRAM once per row block).
constexpr int RASTER_ROWS = 8;   // default group height (BAKRON_TC_RASTER overrides it)

// K tiles of band block (rb, cb): stage 1 those I' with some (I', J') in S1,
// J' in the column block, I' <= I; stage 2 from where stage 1's M coverage
// of these rows starts (M tiles of real rows below k - I are exact zeros
// there); column bands the tile columns of S1, the same for every block.
__device__ __forceinline__ void band_k_range(const TcParams& P, int rb, int cb, int& k0, int& nk) {
  if (P.mode == MODE_COLS) {
    k0 = P.k;
    nk = P.h - P.k;
    return;
  }
  const int I0 = 4 * rb, Ilast = min(I0 + 3, P.Mt - 1);
  const int J0 = 4 * cb;
  if (P.mode == MODE_STAGE1) {
    const int ilo = max(0, P.k - (J0 + 3));
    const int ihi = min(I0 + 3, P.h - 1 - J0);
    k0 = ilo;
    nk = ihi >= ilo ? ihi - ilo + 1 : 0;
    return;
  }
  const int jlo = max(0, P.k - Ilast);
  const int jhi = min(J0 + 3, P.h - 1);
  k0 = jlo;
  nk = jhi >= jlo ? jhi - jlo + 1 : 0;
}

// Returns false if the block has no work at all (beyond its row's span).
__device__ __forceinline__ bool block_of(const TcParams& P, Block& b) {
  // the blocks with the longest K ranges first (they sit at high rows, and
  // in stage 2 at high columns): less of a tail when the grid runs in waves
  int bx = (int)blockIdx.x, by = (int)blockIdx.y;
  if (P.mode != MODE_DENSE && P.mode != MODE_GRAM) {
    const int W = (int)gridDim.x, H = (int)gridDim.y;
    const int R = P.raster > 0 ? P.raster : RASTER_ROWS;
    const int L = by * W + bx, grp = L / (R * W), in = L - grp * R * W;
    const int gh = min(R, H - grp * R);   // rows of this group
    by = grp * R + in % gh;
    bx = in / gh;
  }
  b.rb = P.row0 + (P.mode == MODE_DENSE ? by : (int)gridDim.y - 1 - by);
  b.own = true;
  if (P.mode == MODE_DENSE) {
    b.cb = blockIdx.x;
    b.k0 = b.ok0 = 0;
    b.nk = b.onk = P.K / BK;
    return true;
  }
  if (P.mode == MODE_GRAM) {
    // block t of the lower triangle, row by row: t = rb (rb + 1) / 2 + cb, cb <= rb
    const int t = blockIdx.x;
    int rb = (int)((sqrtf(8.f * (float)t + 1.f) - 1.f) * 0.5f);
    while ((rb + 1) * (rb + 2) / 2 <= t) ++rb;
    while (rb * (rb + 1) / 2 > t) --rb;
    b.rb = rb;
    b.cb = t - rb * (rb + 1) / 2;
    b.k0 = b.ok0 = 0;
    b.nk = b.onk = P.K / BK;   // K stages; the bf16 variant's K counts 128-byte rows of 64
    return true;
  }
  int cb_lo, cb_hi;
  if (!band_row_span(P.mode, P.k, P.h, P.l, P.Mt, P.Nt, b.rb, cb_lo, cb_hi)) return false;
  b.cb = P.mode == MODE_STAGE2 ? cb_hi - bx : cb_lo + bx;
  if (b.cb > cb_hi || b.cb < cb_lo) return false;
  band_k_range(P, b.rb, b.cb, b.k0, b.nk);
  b.ok0 = b.k0;
  b.onk = b.nk;
  b.own = true;
  return true;
}

// Pairs: clusters of two CTAs along x; CTA `rank` of the cluster at grid
// position (blockIdx.x / 2, blockIdx.y) takes row block base + rank; both
// CTAs take the same column block and run the union of their K ranges (this
// CTA's A is zero outside its own).  The decision that the pair has work is
// the same in both CTAs.
__device__ __forceinline__ bool block_of_pair(const TcParams& P, int rank, Block& b) {
  int bx = (int)blockIdx.x >> 1, by = (int)blockIdx.y;
  const int W = (int)gridDim.x >> 1, H = (int)gridDim.y;
  if (P.mode == MODE_DENSE) {
    b.rb = 2 * by + rank;
    b.cb = bx;
    b.k0 = b.ok0 = 0;
    b.nk = b.onk = P.K / BK;
    b.own = true;
    return true;
  }
  {
    const int R = max(1, (P.raster > 0 ? P.raster : RASTER_ROWS) / 2);   // pairs per group
    const int L = by * W + bx, grp = L / (R * W), in = L - grp * R * W;
    const int gh = min(R, H - grp * R);
    by = grp * R + in % gh;
    bx = in / gh;
  }
  const int base = P.row0 + 2 * (H - 1 - by);
  int lo0 = 0, hi0 = -1, lo1 = 0, hi1 = -1;
  const bool v0 = band_row_span(P.mode, P.k, P.h, P.l, P.Mt, P.Nt, base, lo0, hi0);
  const bool v1 = band_row_span(P.mode, P.k, P.h, P.l, P.Mt, P.Nt, base + 1, lo1, hi1);
  if (!v0 && !v1) return false;
  const int cb_lo = v0 && v1 ? min(lo0, lo1) : (v0 ? lo0 : lo1);
  const int cb_hi = v0 && v1 ? max(hi0, hi1) : (v0 ? hi0 : hi1);
  b.cb = P.mode == MODE_STAGE2 ? cb_hi - bx : cb_lo + bx;
  if (b.cb > cb_hi || b.cb < cb_lo) return false;
  const bool s0 = v0 && lo0 <= b.cb && b.cb <= hi0, s1 = v1 && lo1 <= b.cb && b.cb <= hi1;
  int k00 = 0, nk0 = 0, k01 = 0, nk1 = 0;
  if (s0) band_k_range(P, base, b.cb, k00, nk0);
  if (s1) band_k_range(P, base + 1, b.cb, k01, nk1);
  const bool w0 = s0 && nk0 > 0, w1 = s1 && nk1 > 0;   // rows with K tiles
  const int u0 = w0 && w1 ? min(k00, k01) : (w0 ? k00 : k01);
  const int u1 = w0 && w1 ? max(k00 + nk0, k01 + nk1) : (w0 ? k00 + nk0 : k01 + nk1);
  b.rb = base + rank;
  b.own = rank ? s1 : s0;
  b.ok0 = rank ? k01 : k00;
  b.onk = rank ? nk1 : nk0;
  b.k0 = w0 || w1 ? u0 : 0;
  b.nk = w0 || w1 ? u1 - u0 : 0;
  return true;
}

// The kernel body, for the tensor maps of one problem (kernel parameters, so
// their addresses are those of the parameters) and its status word.
template <int V>
__device__ __forceinline__ void tc_body(const CUtensorMap& mapA2, const CUtensorMap& mapB2,
                                        const CUtensorMap& mapBh, const CUtensorMap& mapBl,
                                        const CUtensorMap& mapOh, const CUtensorMap& mapOl,
                                        const TcParams& P, int* status) {
  using RG = Ring<V>;
  constexpr bool pair = RG::pair;
  constexpr int NST = RG::stages;
  constexpr uint32_t SB = RG::stage_bytes;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte alignment for the 128-byte swizzle atoms
  unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* bars = (uint64_t*)(smem + NST * SB);
  uint64_t* full = bars;                 // [NST] smem stage loaded
  uint64_t* empty = bars + NST;          // [NST] slot read by its MMAs (kgroup > 1 only;
                                         // otherwise the slot's accF commit frees it)
  uint64_t* accum = bars + 2 * NST;      // [1] every MMA of the CTA complete
  uint64_t* accF = accum + 1;            // [NACC] accumulator holds a finished K stage
  uint64_t* accE = accum + 1 + NACC;     // [NACC] accumulator read out by the epilogue
  uint32_t* tmem_slot = (uint32_t*)(accum + 1 + 2 * NACC);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // pairs: rank 0 (the leader) issues the MMAs; the loads of both CTAs count
  // on the leader's `full` barriers, the epilogues of both on its `accE`
  const int rank = pair ? (int)cluster_rank() : 0;
  Block blk;
  bool has_block;
  if constexpr (pair) has_block = block_of_pair(P, rank, blk);
  else has_block = block_of(P, blk);
  if (!has_block) {          // uniform over the CTA (and the pair): nothing allocated yet
    pdl_wait();
    pdl_trigger();
    return;
  }

  if (threadIdx.x == 32) {   // descriptors into the cache while the previous kernel runs
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapA2)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapB2)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapBh)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapBl)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapOh)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapOl)) : "memory");
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) {
      mbar_init(&full[s], pair && rank == 0 ? 2 : 1);   // leader: its producer and the peer's
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    for (int a = 0; a < NACC; ++a) {
      mbar_init(&accF[a], 1);
      // lane 0 of each epilogue warp (of both CTAs at the leader)
      mbar_init(&accE[a], pair && rank == 0 ? 2 * EPI_WARPS : EPI_WARPS);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    if constexpr (pair) {   // one warp of each CTA of the pair, same columns in both
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  if constexpr (pair) cluster_sync_all();   // both CTAs' barriers initialised
  else __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  // the leader's barriers in the cluster's shared window (pairs)
  uint32_t cfull0 = 0, caccE0 = 0;
  if constexpr (pair) {
    cfull0 = at_rank0(full);
    caccE0 = at_rank0(accE);
  }
  // The factor operand (stage 1: A = L^B; stage 2: B = L^A) is read-only
  // during the solve: its part of the first ring slots is loaded before the
  // wait for the previous kernel, whose output (E^T or M) is the other one.
  // a wait that ran out stops both CTAs of a pair
  auto abort_all = [&]() {
    *abort_flag = 1;
    if constexpr (pair) st_peer_flag((const void*)abort_flag, rank);
  };
  const int npre = blk.nk < NST ? blk.nk : NST;
  const bool a_static = P.mode != MODE_STAGE2 && P.mode != MODE_COLS;
  constexpr bool bf16_ops = V == V_GRAM_BF16;
  // pairs: this CTA's A is zero (a fully out-of-range box) outside its own K
  // range; its half of B is rows 64 * rank .. of the column block
  auto a_row = [&](int kt) -> int {
    if (!pair) return blk.rb * BM;
    return (blk.own && kt >= blk.ok0 && kt < blk.ok0 + blk.onk) ? blk.rb * BM : -BM;
  };
  const int b_row = pair ? blk.cb * BN + BN_HALF * rank : blk.cb * BN;
  if (warp == 0 && lane == 0) {
    for (int i = 0; i < npre; ++i) {
      unsigned char* st = smem + i * SB;
      const int kt = blk.k0 + i;
      if constexpr (bf16_ops) {
        mbar_expect_tx_only(&full[i], TILE_BYTES);
        tma_load_2d(st, &mapA2, &full[i], kt * 2 * BK, blk.rb * BM);
        continue;
      }
      if constexpr (pair) {
        const uint32_t cb = cfull0 + (uint32_t)(i * 8);
        cmbar_expect_tx_only(cb, a_static ? 2 * TILE_BYTES : 2 * RG::b_plane);
        if (a_static)
          tma_load_pair_c2(st, &mapA2, cb, kt * BK, a_row(kt));
        else
          tma_load_pair_c2(st + 2 * TILE_BYTES, &mapB2, cb, kt * BK, b_row);
        continue;
      }
      mbar_expect_tx_only(&full[i], 2 * TILE_BYTES);
      if (a_static)
        tma_load_pair(st, &mapA2, &full[i], kt * BK, blk.rb * BM);
      else
        tma_load_pair(st + 2 * TILE_BYTES, &mapB2, &full[i], kt * BK, blk.cb * BN);
    }
  }
  // the rest waits for the previous kernel
  pdl_wait();
  pdl_trigger();
  stamp_begin(P.stamp);
  const long long drain = 4000000000LL;   // ~2 s at 2 GHz: wind-down bound
  const int nk = blk.nk;
  constexpr int kgroup = V == V_GRAM_BF16 ? GRAM_KGROUP : (V == V_BAND ? BAND_KGROUP : 1);
  const int ngroups = (nk + kgroup - 1) / kgroup;   // accumulator hand-overs

  if (warp == 0) {
    // ---------------------------------------------------------- producer
    int issued = 0;
    bool aborted = false;
    for (int i = 0; i < nk; ++i) {
      const int s = i % NST;
      bool ok = true;
      // slot s was last read by the MMAs of stage j = i - NST, which are
      // complete when their accumulator's commit arrives (accF); that barrier
      // cannot have moved on to stage j + NACC yet, which needs this load
      if (lane == 0 && i >= NST) {
        const int j = i - NST;
        if constexpr (kgroup > 1)
          ok = mbar_wait(&empty[s], (uint32_t)(j / NST) & 1u, P.spin_cycles);
        else
          ok = mbar_wait(&accF[j % NACC], (uint32_t)(j / NACC) & 1u, P.spin_cycles);
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok || *abort_flag) {
        if (lane == 0 && !ok) { raise_status(status, BAKRON_ERR_TIMEOUT); abort_all(); }
        // slots loaded in part before the wait: arrive, so that their phase
        // completes once those copies land (the drain below waits for them)
        if (lane == 0) {
          for (int j = i; j < npre; ++j) {
            if constexpr (pair) cmbar_arrive(cfull0 + (uint32_t)(j * 8));
            else mbar_arrive(&full[j]);
          }
        }
        aborted = true;
        break;
      }
      unsigned char* st = smem + s * SB;
      // planes of the slot: A hi, A lo, B hi, B lo (a pair lands as hi then lo)
      unsigned char *a_hi = st, *b_hi = st + 2 * TILE_BYTES, *b_lo = b_hi + RG::b_plane;
      const int kt = blk.k0 + i;            // K tile index (32 wide)
      const bool pre = i < npre;            // the factor operand is already on its way
      if constexpr (bf16_ops) {             // one bf16 box per operand, 64 of K
        if (lane == 0) {
          mbar_expect_tx(&full[s], pre ? TILE_BYTES : 2 * TILE_BYTES);
          if (!pre) tma_load_2d(a_hi, &mapA2, &full[s], kt * 2 * BK, blk.rb * BM);
          tma_load_2d(b_hi, &mapB2, &full[s], kt * 2 * BK, blk.cb * BN);
        }
        __syncwarp();
        issued = i + 1;
        continue;
      }
      const bool load_a = !(pre && a_static), load_b = !(pre && !a_static);
      if constexpr (pair) {
        // every box lands in full (an out-of-range one as zeros), so the
        // byte count does not depend on the band
        if (lane == 0) {
          const uint32_t cb = cfull0 + (uint32_t)(s * 8);
          cmbar_arrive_expect_tx(cb, (load_a ? 2 * TILE_BYTES : 0u) +
                                         (load_b ? 2 * RG::b_plane : 0u));
          if (load_a) tma_load_pair_c2(a_hi, &mapA2, cb, kt * BK, a_row(kt));
          if (load_b) {
            unsigned valid = 3u;            // stage 1: this half's two sub-tiles in the band
            if (P.mode == MODE_STAGE1) {
              valid = 0;
              for (int sub = 0; sub < 2; ++sub) {
                const int Jp = 4 * blk.cb + 2 * rank + sub;
                if (Jp < P.Nt && kt < P.Mt && kt + Jp >= P.k && kt + Jp < P.h) valid |= 1u << sub;
              }
            }
            if (valid == 3u) {
              tma_load_pair_c2(b_hi, &mapB2, cb, kt * BK, b_row);   // b_lo follows
            } else {
              for (int sub = 0; sub < 2; ++sub) {
                const int y = (valid & (1u << sub)) ? b_row + 32 * sub : -32;
                tma_load_2d_c2(b_hi + sub * 4096, &mapBh, cb, kt * BK, y);
                tma_load_2d_c2(b_lo + sub * 4096, &mapBl, cb, kt * BK, y);
              }
            }
          }
        }
        __syncwarp();
        issued = i + 1;
        continue;
      }
      uint32_t bytes = load_a ? 2 * TILE_BYTES : 0u;   // A hi + A lo
      unsigned valid = 0xF;                 // stage 1: B sub-tiles in the band
      if (P.mode == MODE_STAGE1) {
        valid = 0;
        for (int sub = 0; sub < 4; ++sub) {
          const int Jp = 4 * blk.cb + sub;
          const bool v = Jp < P.Nt && kt < P.Mt && kt + Jp >= P.k && kt + Jp < P.h;
          if (v) valid |= 1u << sub;
        }
        // zero-fill the sub-tiles outside the band (4 KiB each, hi and lo)
        for (int sub = 0; sub < 4; ++sub) {
          if (valid & (1u << sub)) continue;
          float4* zh = reinterpret_cast<float4*>(b_hi + sub * 4096);
          float4* zl = reinterpret_cast<float4*>(b_lo + sub * 4096);
          for (int e = lane; e < 256; e += 32) {
            zh[e] = make_float4(0.f, 0.f, 0.f, 0.f);
            zl[e] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        bytes += 2u * 4096u * (uint32_t)__popc(valid);
      } else if (load_b) {
        bytes += 2 * TILE_BYTES;
      }
      if (lane == 0) {
        mbar_expect_tx(&full[s], bytes);
        if (load_a) tma_load_pair(a_hi, &mapA2, &full[s], kt * BK, blk.rb * BM);   // a_lo follows
        if (!load_b) {
        } else if (P.mode == MODE_STAGE1 && valid == 0xFu) {   // inside the band: one box, both planes
          tma_load_pair(b_hi, &mapB2, &full[s], kt * BK, blk.cb * BN);
        } else if (P.mode == MODE_STAGE1) {
          for (int sub = 0; sub < 4; ++sub) {
            if (!(valid & (1u << sub))) continue;
            const int y = (4 * blk.cb + sub) * 32;
            tma_load_2d(b_hi + sub * 4096, &mapBh, &full[s], kt * BK, y);
            tma_load_2d(b_lo + sub * 4096, &mapBl, &full[s], kt * BK, y);
          }
        } else {
          tma_load_pair(b_hi, &mapB2, &full[s], kt * BK, blk.cb * BN);   // b_lo follows
        }
      }
      __syncwarp();
      issued = i + 1;
    }
    // drain: every copy this warp issued has landed before the CTA winds down
    if (lane == 0) {
      // pairs: after an abort a leader's phase may lack the peer's arrival,
      // and the peer cannot watch the leader's barriers; copies in flight land
      // within microseconds, so both wait about a millisecond instead
      constexpr long long kPairSettle = 2000000LL;
      if (pair && (rank != 0 || *abort_flag)) {
        if (aborted || *abort_flag) {
          const long long t0 = clock64();
          while (clock64() - t0 < kPairSettle) __nanosleep(1000);
        }
      } else {
        const int last = issued > npre ? issued : npre;
        const int first = last > NST ? last - NST : 0;
        for (int i = first; i < last; ++i) {
          if (!mbar_wait(&full[i % NST], (uint32_t)(i / NST) & 1u, drain))
            raise_status(status, BAKRON_ERR_TIMEOUT);
        }
      }
    }
  } else if (warp == 1) {
    // --------------------------------------------------------- MMA issuer
    // Each group of kgroup K stages (one stage in the band products, four of
    // exact bf16 products in the Gram) accumulates afresh into accumulator
    // (group mod NACC); the epilogue adds the groups in fp32 registers.  The
    // tensor core's accumulation is not round-to-nearest, and its error grows
    // with the number of MMAs summed in place; restarting every group bounds it.
    if (lane == 0 && pair && rank != 0) {
      // the peer: the leader's MMAs write this CTA's TMEM and read its shared
      // memory; its last commit arrives here too once they have completed
      if (nk == 0) mbar_arrive(accum);
      if (!mbar_wait(accum, 0, drain)) raise_status(status, BAKRON_ERR_TIMEOUT);
    } else if (lane == 0) {
      const uint32_t idesc = idesc_tf32(pair ? 2 * BM : BM, BN), idesc_b = idesc_bf16(BM, BN);
      const uint64_t desc0 = smem_desc(smem_u32(smem));   // stage 0, A hi, K step 0
      for (int i = 0; i < nk; ++i) {
        const int s = i % NST;
        const uint32_t ph = (uint32_t)(i / NST) & 1u;
        const int g = i / kgroup, a = g % NACC;     // accumulator group of this slot
        const bool first = i % kgroup == 0;
        const bool last = i % kgroup == kgroup - 1 || i == nk - 1;
        // accumulator a was last used by group g - NACC: wait until it was read
        // out (the producer's and the epilogue's aborts surface here as time-outs)
        bool ok;
        if constexpr (pair)
          ok = mbar_wait_cluster(&full[s], ph, P.spin_cycles) &&
               (!first || g < NACC ||
                mbar_wait_cluster(&accE[a], (uint32_t)(g / NACC - 1) & 1u, P.spin_cycles));
        else
          ok = mbar_wait(&full[s], ph, P.spin_cycles) &&
               (!first || g < NACC ||
                mbar_wait(&accE[a], (uint32_t)(g / NACC - 1) & 1u, P.spin_cycles));
        if (!ok) {
          raise_status(status, BAKRON_ERR_TIMEOUT);
          abort_all();
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // descriptors of this stage's four planes; K steps of 32 bytes add 2 to
        // the start-address field (16-byte units, no carry within a stage)
        const uint64_t dah = desc0 + (uint64_t)((s * SB) >> 4);
        const uint64_t dal = dah + (TILE_BYTES >> 4), dbh = dah + (2 * TILE_BYTES >> 4),
                       dbl = dbh + (RG::b_plane >> 4);
        const uint32_t d = tmem + (uint32_t)(a * BN);
        if constexpr (bf16_ops) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)            // 16 bf16 = 32 bytes along K per MMA
            mma_bf16(d, dah + 2 * kk, dbh + 2 * kk, idesc_b, (kk > 0 || !first) ? 1u : 0u);
        } else if constexpr (pair) {
#pragma unroll
          for (int kk = 0; kk < BK / 8; ++kk) {
            const uint64_t o = (uint64_t)(2 * kk);
            mma_tf32_pair(d, dah + o, dbh + o, idesc, (kk > 0 || !first) ? 1u : 0u);
            mma_tf32_pair(d, dah + o, dbl + o, idesc, 1u);
            mma_tf32_pair(d, dal + o, dbh + o, idesc, 1u);
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < BK / 8; ++kk) {
            const uint64_t o = (uint64_t)(2 * kk);   // 8 tf32 = 32 bytes along K inside the swizzle row
            mma_tf32(d, dah + o, dbh + o, idesc, (kk > 0 || !first) ? 1u : 0u);
            if (V == V_BAND || !P.b_exact) mma_tf32(d, dah + o, dbl + o, idesc, 1u);
            if (V == V_BAND || !P.a_exact) mma_tf32(d, dal + o, dbh + o, idesc, 1u);
          }
        }
        if constexpr (pair) {
          if (last) mma_commit_pair(&accF[a]);   // both CTAs: the sum, and the slot
        } else {
          if constexpr (kgroup > 1) mma_commit(&empty[s]);   // the slot back to the producer
          if (last) mma_commit(&accF[a]);  // the group's sum to the epilogue (kgroup 1: and the slot)
        }
      }
      if (nk > 0) {  // tracks every MMA issued above
        if constexpr (pair) mma_commit_pair(accum);
        else mma_commit(accum);
      } else {
        mbar_arrive(accum);
      }
      // wind-down guard: all issued MMAs complete before anyone frees TMEM
      if (!mbar_wait(accum, 0, drain)) raise_status(status, BAKRON_ERR_TIMEOUT);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;                 // TMEM lane quarter of this warp
    const int c0 = ((warp - 2) >> 2) * EPI_COLS;   // its half of the 128 columns
    const int row = q * 32 + lane;          // row inside the 128 x 128 block
    float acc[EPI_COLS];
#pragma unroll
    for (int u = 0; u < EPI_COLS; ++u) acc[u] = 0.f;
    bool write = blk.own;
    for (int i = 0; i < ngroups; ++i) {
      const int a = i % NACC;
      // one lane waits; the decision is warp-uniform (tcgen05.ld is warp-collective)
      int ok = 1;
      if (lane == 0) {
        ok = mbar_wait(&accF[a], (uint32_t)(i / NACC) & 1u, P.spin_cycles) ? 1 : 0;
        if (!ok) { raise_status(status, BAKRON_ERR_TIMEOUT); abort_all(); }
        if (*abort_flag) ok = 0;
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) { write = false; break; }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t ta = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(a * BN + c0);
      uint32_t r0[32], r1[32];
      tmem_ld32(ta, r0);
      tmem_ld32(ta + 32, r1);
      tmem_wait_ld();
#pragma unroll
      for (int u = 0; u < 32; ++u) {
        acc[u] += __uint_as_float(r0[u]);
        acc[32 + u] += __uint_as_float(r1[u]);
      }
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) {
        if constexpr (pair) cmbar_arrive(caccE0 + (uint32_t)(a * 8));
        else mbar_arrive(&accE[a]);
      }
    }
    if (P.mode == MODE_GRAM) {
      // entry (gi, gj <= gi) and its mirror (gj, gi); for a fixed u the warp's
      // 32 lanes hold 32 consecutive gi, so the mirror stores are coalesced
      const int64_t gi = (int64_t)blk.rb * BM + row;
      const int64_t gj0 = (int64_t)blk.cb * BN + c0;
      if (write && gi < P.dreal) {
#pragma unroll
        for (int u = 0; u < EPI_COLS; ++u) {
          const int64_t gj = gj0 + u;
          if (gj > gi) continue;          // also keeps gj < dreal
          const float v = P.alpha * acc[u];
          float* p = P.out_hi + gi * P.ldo + gj;
          *p = P.beta == 0.f ? v : fmaf(P.beta, *p, v);
          if (gj < gi) {
            float* q2 = P.out_hi + gj * P.ldo + gi;
            *q2 = P.beta == 0.f ? v : fmaf(P.beta, *q2, v);
          }
        }
      }
    } else if (P.mode == MODE_DENSE) {
      const int64_t gi = (int64_t)blk.rb * BM + row;
#pragma unroll
      for (int c = 0; c < EPI_COLS / 32; ++c) {
        if (!write) break;
        const float* v = &acc[c * 32];
        const int64_t gj = (int64_t)blk.cb * BN + c0 + c * 32;
        float4* o = reinterpret_cast<float4*>(P.out_hi + gi * P.ldo + gj);
#pragma unroll
        for (int u = 0; u < 8; ++u) o[u] = make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
      }
    } else {
      // Every MMA has completed (the last accumulator was committed after
      // them), so the ring is free: stage the block as 32-column boxes of 128
      // rows, box (plane, c) at smem + (plane * 4 + c) * 16 KiB, 16-byte chunk
      // u of row r at chunk u ^ (r & 7) (the 128-byte swizzle of the maps).
      if (write) {
#pragma unroll
        for (int c = 0; c < EPI_COLS / 32; ++c) {
          const int cb32 = (c0 >> 5) + c;     // 32-column box of this chunk
          const float* v = &acc[c * 32];
          unsigned char* rowh = smem + cb32 * TILE_BYTES + row * 128;
          unsigned char* rowl = rowh + 4 * TILE_BYTES;
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int off = ((u ^ (row & 7)) << 4);
            if (P.mode == MODE_STAGE1) {
              float hi[4], lo[4];
#pragma unroll
              for (int w2 = 0; w2 < 4; ++w2) {
                hi[w2] = tf32_hi(v[4 * u + w2]);
                lo[w2] = v[4 * u + w2] - hi[w2];
              }
              *reinterpret_cast<float4*>(rowh + off) = make_float4(hi[0], hi[1], hi[2], hi[3]);
              *reinterpret_cast<float4*>(rowl + off) = make_float4(lo[0], lo[1], lo[2], lo[3]);
            } else {
              *reinterpret_cast<float4*>(rowh + off) =
                  make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
            }
          }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // visible to the TMA unit
      }
      asm volatile("bar.sync 2, %0;" ::"n"(EPI_WARPS * 32) : "memory");   // the epilogue warps
      if (warp == 2 && lane == 0 && !*abort_flag && blk.own) {
        const int x0 = blk.cb * BN, y0 = blk.rb * BM;
        if (P.mode == MODE_STAGE1) {
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            tma_store_2d(&mapOh, smem + c * TILE_BYTES, x0 + 32 * c, y0);
            tma_store_2d(&mapOl, smem + (4 + c) * TILE_BYTES, x0 + 32 * c, y0);
          }
        } else if (blk.onk > 0) {
          // X += the block's tiles that lie in S2 (32 x 32 boxes: rows 32 ti
          // .. of box c start 4 KiB apart, whole swizzle periods)
          for (int ti = 0; ti < 4; ++ti) {
            for (int c = 0; c < 4; ++c) {
              const int I = 4 * blk.rb + ti, J = 4 * blk.cb + c;
              if (I >= P.Mt || J >= P.Nt) continue;
              if (P.mode == MODE_COLS ? (J < P.h || J >= P.l) : (I + J < P.h || I + J >= P.l))
                continue;
              tma_reduce_add_2d(&mapOh, smem + c * TILE_BYTES + ti * 4096, 32 * J, 32 * I);
            }
          }
        }
        bulk_commit_and_wait();   // complete before the CTA (and its shared memory) goes
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  // pairs: neither CTA leaves (nor frees TMEM) while the other may still
  // signal its barriers or use its shared memory
  if constexpr (pair) cluster_sync_all();
  else __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  stamp_end(P.stamp);
  if (warp == 1) {
    if constexpr (pair)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                   "r"(TMEM_COLS)
                   : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                   "r"(TMEM_COLS)
                   : "memory");
  }
}

template <int V>
__global__ void __launch_bounds__(THREADS, 1)
k_tc_band(const __grid_constant__ CUtensorMap mapA2, const __grid_constant__ CUtensorMap mapB2,
          const __grid_constant__ CUtensorMap mapBh, const __grid_constant__ CUtensorMap mapBl,
          const __grid_constant__ CUtensorMap mapOh, const __grid_constant__ CUtensorMap mapOl,
          const TcParams P) {
  tc_body<V>(mapA2, mapB2, mapBh, mapBl, mapOh, mapOl, P, P.status);
}

// One band stage of up to TC_MAX_HEADS problems of one shape in one launch
// (blockIdx.z = problem): each problem's six tensor maps and status word
// (about 25 KB of kernel parameters in all, within the 32 KB limit).
constexpr int TC_MAX_HEADS = 32;
struct TcHeads {
  CUtensorMap maps[TC_MAX_HEADS][6];   // A2, B2, Bh, Bl, Oh, Ol per problem
  int* status[TC_MAX_HEADS];
  TcParams P;
};

__global__ void __launch_bounds__(THREADS, 1) k_tc_heads(const __grid_constant__ TcHeads T) {
  const CUtensorMap* m = T.maps[blockIdx.z];
  tc_body<V_BAND>(m[0], m[1], m[2], m[3], m[4], m[5], T.P, T.status[blockIdx.z]);
}

// ------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encode() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  });
  return g_encode != nullptr;
}

// 2-D fp32 row-major matrix (rows x cols, row stride ld elements), box of
// 32 columns (128 bytes, one swizzle row) by box_rows rows, 128-byte swizzle.
bool make_map(CUtensorMap* map, const float* base, int64_t rows, int64_t cols, int64_t ld,
              int box_rows) {
  if (!get_encode()) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * 4)};
  cuuint32_t box[2] = {32u, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1u, 1u};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, (void*)base, dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The hi/lo pair of a 2-D fp32 matrix whose lo plane starts plane_bytes
// after its hi plane, as a rank-3 tensor (columns, rows, plane): boxes of 32
// columns x box_rows rows x both planes, 128-byte swizzle.
bool make_map_pair(CUtensorMap* map, const float* hi, const float* lo, int64_t rows, int64_t cols,
                   int64_t ld, int box_rows) {
  if (!get_encode()) return false;
  const int64_t plane_bytes = (const char*)lo - (const char*)hi;
  if (plane_bytes < rows * ld * 4 || plane_bytes % 16) return false;
  cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, 2u};
  cuuint64_t strides[2] = {(cuuint64_t)(ld * 4), (cuuint64_t)plane_bytes};
  cuuint32_t box[3] = {32u, (cuuint32_t)box_rows, 2u};
  cuuint32_t estr[3] = {1u, 1u, 1u};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, (void*)hi, dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 2-D bf16 row-major matrix (rows x cols, row stride ld elements), box of 64
// columns (128 bytes, one swizzle row) by box_rows rows, 128-byte swizzle.
bool make_map_bf16(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld,
                   int box_rows) {
  if (!get_encode() || (ld * 2) % 16) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * 2)};
  cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1u, 1u};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)base, dims, strides,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool g_attr_done = false;
std::mutex g_attr_mu;

cudaError_t ensure_attr() {
  std::lock_guard<std::mutex> lk(g_attr_mu);
  if (g_attr_done) return cudaSuccess;
  cudaError_t e =
      cudaFuncSetAttribute(k_tc_band<V_BAND>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           SMEM_BYTES);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_tc_band<V_GRAM_TF32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_tc_band<V_GRAM_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_tc_band<V_PAIR>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             PAIR_SMEM_BYTES);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_tc_heads, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e == cudaSuccess) g_attr_done = true;
  return e;
}

// The paired kernel: clusters of two CTAs along x, with programmatic
// dependent launch like every other kernel of the solve (pdl = false: a
// plain launch, for the diagnostic GEMM).
template <typename... Args>
cudaError_t launch_pair(dim3 grid, cudaStream_t s, bool pdl, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = PAIR_SMEM_BYTES;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, k_tc_band<V_PAIR>, args...);
}

// hi/lo split of a dense matrix (diagnostic GEMM only)
__global__ void k_split(const float* src, int64_t count, float* hi, float* lo) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= count) return;
  const float v = src[i], h = tf32_hi(v);
  hi[i] = h;
  lo[i] = v - h;
}

// Gram operands: samples t0 .. t0 + kc of X (k x d, row stride ldx, fp32 or
// bf16) transposed into the K-major planes T = X^T (dp x kc, zeros past k and
// d), split as hi + lo; with weights, also WT = (diag(w) X)^T, the product
// w_t x_ti rounded once to fp32 before the split.  32 x 32 tiles through
// shared memory: coalesced reads along features, writes along samples.
__global__ void k_gram_split(const void* X, int xdt, int k, int d, int64_t ldx, int t0, int kc,
                             const float* w, float* Th, float* Tl, float* Wh, float* Wl) {
  __shared__ float tile[32][33];
  __shared__ float wt[32];
  const int tx = threadIdx.x, ty = threadIdx.y;     // 32 x 8
  const int tb = blockIdx.x * 32, ib = blockIdx.y * 32;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int t = t0 + tb + ty + 8 * r, i = ib + tx;
    float v = 0.f;
    if (t < k && i < d) {
      const int64_t o = (int64_t)t * ldx + i;
      v = xdt == BAKRON_BF16 ? __bfloat162float(((const __nv_bfloat16*)X)[o])
                             : ((const float*)X)[o];
    }
    tile[ty + 8 * r][tx] = v;
  }
  if (w && ty == 0) wt[tx] = (t0 + tb + tx < k) ? w[t0 + tb + tx] : 0.f;
  __syncthreads();
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int i = ib + ty + 8 * r, tc = tb + tx;
    const int64_t o = (int64_t)i * kc + tc;
    const float v = tile[tx][ty + 8 * r], h = tf32_hi(v);
    Th[o] = h;
    Tl[o] = v - h;
    if (w) {
      const float u = wt[tx] * v, uh = tf32_hi(u);
      Wh[o] = uh;
      Wl[o] = u - uh;
    }
  }
}

// bf16 samples t0 .. t0 + kc of X (k x d, row stride ldx) transposed into
// the K-major bf16 plane T = X^T (dp x kc, zeros past k and d): the operand of
// the kind::f16 Gram, exact (no split).  64 x 64 tiles through shared memory,
// 16-byte vectors both ways: a load is 8 features of one sample (when X and
// ldx allow 16-byte alignment and the 8 lie inside d; else element by
// element), a store 8 samples of one feature (always whole: dp and kc are
// multiples of 64).  A warp reads 4 rows of 128 bytes and stores 32 rows'
// 16-byte pieces; its shared-memory gathers read one 64-byte row segment.
constexpr int TR_TILE = 64, TR_LD = 72;   // row stride 144 B: 16-byte aligned rows

__global__ void __launch_bounds__(256)
    k_gram_transpose_bf16(const __nv_bfloat16* X, int k, int d, int64_t ldx, int t0, int kc,
                          int vec_ok, __nv_bfloat16* T) {
  __shared__ __align__(16) __nv_bfloat16 tile[TR_TILE][TR_LD];
  const int tb = blockIdx.x * TR_TILE, ib = blockIdx.y * TR_TILE;
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int c = threadIdx.x + 256 * r;          // 512 chunks of 8 features
    const int tr = c >> 3, i0 = ib + 8 * (c & 7);
    const int t = t0 + tb + tr;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (t < k) {
      const __nv_bfloat16* src = X + (int64_t)t * ldx + i0;
      if (vec_ok && i0 + 8 <= d) {
        v = *reinterpret_cast<const uint4*>(src);
      } else {
        __align__(16) __nv_bfloat16 e[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) e[j] = (i0 + j < d) ? src[j] : __float2bfloat16(0.f);
        v = *reinterpret_cast<const uint4*>(e);
      }
    }
    *reinterpret_cast<uint4*>(&tile[tr][8 * (c & 7)]) = v;
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int c = threadIdx.x + 256 * r;          // 512 chunks of 8 samples
    const int ir = c & 63, tc = c >> 6;
    __align__(16) __nv_bfloat16 e[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) e[j] = tile[8 * tc + j][ir];
    *reinterpret_cast<uint4*>(T + (int64_t)(ib + ir) * kc + tb + 8 * tc) =
        *reinterpret_cast<const uint4*>(e);
  }
}

// |y_t|^2 per row (warp per row, fp32, lane-strided partial sums then a
// butterfly): the one-step Shampoo weight tr(b_t^T b_t) of a vector sample.
__global__ void k_sqnorms(const void* Y, int ydt, int k, int d, int64_t ldy, float* out) {
  const int64_t row = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= k) return;
  float acc = 0.f;
  for (int j = lane; j < d; j += 32) {
    const int64_t o = row * ldy + j;
    const float v = ydt == BAKRON_BF16 ? __bfloat162float(((const __nv_bfloat16*)Y)[o])
                                       : ((const float*)Y)[o];
    acc = fmaf(v, v, acc);
  }
  for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) out[row] = acc;
}

}  // namespace

long long spin_cycles_from_env() {
  const char* e = getenv("BAKRON_SPIN_CYCLES");
  if (e && *e) {
    long long v = atoll(e);
    if (v >= 0) return v;
  }
  return 4000000000LL;  // ~2 s at 2 GHz
}

bool tc_band_maps(TcMaps& maps, const TcOperands& op) {
  // stage 1: A = L^B (mp x mp), B = E^T (np x mp) in 32-row boxes
  // stage 2: A = M (mp x np), B = L^A (np x np)
  bool ok = true;
  ok &= make_map_pair(&maps.LB2, op.LBH, op.LBL, op.mp, op.mp, op.mp, BM);
  ok &= make_map(&maps.Eth, op.EtH, op.np, op.mp, op.mp, 32);
  ok &= make_map(&maps.Etl, op.EtL, op.np, op.mp, op.mp, 32);
  ok &= make_map_pair(&maps.Et2, op.EtH, op.EtL, op.np, op.mp, op.mp, BN);
  ok &= make_map(&maps.Mh, op.MH, op.mp, op.np, op.np, BM);
  ok &= make_map(&maps.Ml, op.ML, op.mp, op.np, op.np, BM);
  ok &= make_map_pair(&maps.M2, op.MH, op.ML, op.mp, op.np, op.np, BM);
  ok &= make_map_pair(&maps.LA2, op.LAH, op.LAL, op.np, op.np, op.np, BN);
  ok &= make_map_pair(&maps.Et2h, op.EtH, op.EtL, op.np, op.mp, op.mp, BN_HALF);   // pairs' B halves
  ok &= make_map_pair(&maps.LA2h, op.LAH, op.LAL, op.np, op.np, op.np, BN_HALF);
  ok &= make_map(&maps.X32, op.X, op.mp, op.np, op.np, 32);   // stage-2 reduce target
  return ok;
}

// Group height of the band stages' launch order (BAKRON_TC_RASTER, read per call).
static int raster_rows() {
  const char* e = getenv("BAKRON_TC_RASTER");
  const int v = e ? atoi(e) : 0;
  return v >= 1 ? v : RASTER_ROWS;
}

// Band stages on CTA pairs (BAKRON_TC_PAIR=1/0, read per call; default kTcPairDefault).
constexpr bool kTcPairDefault = false;
bool tc_pair_on() {
  const char* e = getenv("BAKRON_TC_PAIR");
  if (e && *e) return atoi(e) != 0;
  return kTcPairDefault;
}

// Pairs: the widest union of column spans over the row-block pairs
// (rlo + 2p, rlo + 2p + 1) of rows [rlo, rhi].
static int pair_width(int mode, int k, int h, int l, int Mt, int Nt, int rlo, int rhi) {
  int width = 0;
  for (int r0 = rlo; r0 <= rhi; r0 += 2) {
    int lo = 1 << 30, hi = -1;
    for (int r = r0; r <= r0 + 1; ++r) {
      int cl, ch;
      if (!band_row_span(mode, k, h, l, Mt, Nt, r, cl, ch)) continue;
      lo = std::min(lo, cl);
      hi = std::max(hi, ch);
    }
    if (hi >= 0) width = std::max(width, hi - lo + 1);
  }
  return width;
}

int tc_band_stage(int stage, const TcMaps& maps, const TcOperands& op, int k, int h, int l,
                  cudaStream_t s, unsigned long long* stamp) {
  BK_CUDA_OK(ensure_attr());
  TcParams P{};
  P.stamp = stamp;
  P.raster = raster_rows();
  P.mode = stage == 1 ? MODE_STAGE1 : MODE_STAGE2;
  P.k = k; P.h = h; P.l = l;
  P.Mt = op.Mt; P.Nt = op.Nt;
  P.out_hi = op.MH; P.out_lo = op.ML; P.X = op.X;
  P.ldo = op.np;
  P.status = op.status;
  P.spin_cycles = spin_cycles_from_env();
  // bounding box of the output blocks with work: rows [rlo, rhi], and the
  // widest row's span of column blocks
  int rlo = -1, rhi = -1, width = 0;
  const int nb_rows = (int)(op.mp / BM);
  for (int rb = 0; rb < nb_rows; ++rb) {
    int cl, ch;
    if (!band_row_span(P.mode, k, h, l, op.Mt, op.Nt, rb, cl, ch)) continue;
    if (rlo < 0) rlo = rb;
    rhi = rb;
    width = std::max(width, ch - cl + 1);
  }
  if (rlo < 0) return BAKRON_OK;   // nothing to do in this stage
  P.row0 = rlo;
  cudaError_t e;
  if (tc_pair_on()) {
    const int pairs = (rhi - rlo) / 2 + 1;
    dim3 pg(2 * pair_width(P.mode, k, h, l, op.Mt, op.Nt, rlo, rhi), pairs);
    if (stage == 1)
      e = launch_pair(pg, s, true, maps.LB2, maps.Et2h, maps.Eth, maps.Etl, maps.Mh, maps.Ml, P);
    else
      e = launch_pair(pg, s, true, maps.M2, maps.LA2h, maps.Eth, maps.Etl, maps.X32, maps.X32, P);
    return BK_CUDA_RC(e);
  }
  dim3 grid(width, rhi - rlo + 1);
  if (stage == 1)
    e = launch_pdl(k_tc_band<V_BAND>, grid, dim3(THREADS), SMEM_BYTES, s, maps.LB2, maps.Et2,
                   maps.Eth,
                   maps.Etl, maps.Mh, maps.Ml, P);
  else   // (the 32-row E^T maps are not read in stage 2)
    e = launch_pdl(k_tc_band<V_BAND>, grid, dim3(THREADS), SMEM_BYTES, s, maps.M2, maps.LA2,
                   maps.Eth,
                   maps.Etl, maps.X32, maps.X32, P);
  return BK_CUDA_RC(e);
}

int tc_band_stage_heads(int stage, int H, const TcMaps* const* maps, int* const* status,
                        const TcOperands& op, int k, int h, int l, cudaStream_t s,
                        unsigned long long* stamp) {
  if (H < 1 || H > TC_MAX_HEADS) return BAKRON_ERR_INVALID_ARG;
  BK_CUDA_OK(ensure_attr());
  static thread_local TcHeads T;   // 25 KB: kept off the stack
  TcParams& P = T.P;
  P = TcParams{};
  P.stamp = stamp;
  P.raster = raster_rows();
  P.mode = stage == 1 ? MODE_STAGE1 : MODE_STAGE2;
  P.k = k; P.h = h; P.l = l;
  P.Mt = op.Mt; P.Nt = op.Nt;
  P.ldo = op.np;
  P.spin_cycles = spin_cycles_from_env();
  int rlo = -1, rhi = -1, width = 0;
  const int nb_rows = (int)(op.mp / BM);
  for (int rb = 0; rb < nb_rows; ++rb) {
    int cl, ch;
    if (!band_row_span(P.mode, k, h, l, op.Mt, op.Nt, rb, cl, ch)) continue;
    if (rlo < 0) rlo = rb;
    rhi = rb;
    width = std::max(width, ch - cl + 1);
  }
  if (rlo < 0) return BAKRON_OK;
  P.row0 = rlo;
  for (int p = 0; p < H; ++p) {
    const TcMaps& m = *maps[p];
    CUtensorMap* d = T.maps[p];
    if (stage == 1) {
      d[0] = m.LB2; d[1] = m.Et2; d[2] = m.Eth; d[3] = m.Etl; d[4] = m.Mh; d[5] = m.Ml;
    } else {
      d[0] = m.M2; d[1] = m.LA2; d[2] = m.Eth; d[3] = m.Etl; d[4] = m.X32; d[5] = m.X32;
    }
    T.status[p] = status[p];
  }
  return BK_CUDA_RC(launch_pdl(k_tc_heads, dim3(width, rhi - rlo + 1, H), dim3(THREADS),
                               SMEM_BYTES, s, T));
}

int tc_cols_stage(const TcMaps& maps, const TcOperands& op, int k, int h, int l, cudaStream_t s,
                  unsigned long long* stamp) {
  BK_CUDA_OK(ensure_attr());
  if (k >= h || h >= l) return BAKRON_OK;
  TcParams P{};
  P.stamp = stamp;
  P.raster = raster_rows();
  P.mode = MODE_COLS;
  P.k = k; P.h = h; P.l = l;
  P.Mt = op.Mt; P.Nt = op.Nt;
  P.out_hi = op.MH; P.out_lo = op.ML; P.X = op.X;
  P.ldo = op.np;
  P.status = op.status;
  P.spin_cycles = spin_cycles_from_env();
  const int rows = (op.Mt + 3) / 4;              // 128-row blocks holding real tiles
  const int cols = (l - 1) / 4 - h / 4 + 1;      // 128-column blocks covering S2
  P.row0 = 0;
  if (tc_pair_on()) {
    const cudaError_t e = launch_pair(dim3(2 * cols, (rows + 1) / 2), s, true, maps.M2,
                                      maps.LA2h, maps.Eth, maps.Etl, maps.X32, maps.X32, P);
    return BK_CUDA_RC(e);
  }
  const cudaError_t e =
      launch_pdl(k_tc_band<V_BAND>, dim3(cols, rows), dim3(THREADS), SMEM_BYTES, s, maps.M2,
                 maps.LA2, maps.Eth, maps.Etl, maps.X32, maps.X32, P);
  return BK_CUDA_RC(e);
}

}  // namespace bakron

using namespace bakron;

extern "C" int bakron_diag_gemm_tf32x3(const float* A, const float* B, float* C, int M, int N,
                                       int K, void* workspace, size_t workspace_bytes,
                                       void* stream) {
  if (!A || !B || !C || !workspace || M <= 0 || N <= 0 || K <= 0) return BAKRON_ERR_INVALID_ARG;
  if (M % BM || N % BN || K % BK) return BAKRON_ERR_INVALID_ARG;
  const size_t need = 256 + size_t(2) * (size_t(M) + N) * K * 4;
  if (workspace_bytes < need) return BAKRON_ERR_WORKSPACE;
  BK_CUDA_OK(ensure_attr());
  cudaStream_t s = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  int* status = (int*)ws;
  float* Ah = (float*)(ws + 256);
  float* Al = Ah + (size_t)M * K;
  float* Bh = Al + (size_t)M * K;
  float* Bl = Bh + (size_t)N * K;
  BK_CUDA_OK(cudaMemsetAsync(status, 0, 256, s));
  k_split<<<(unsigned)(((int64_t)M * K + 255) / 256), 256, 0, s>>>(A, (int64_t)M * K, Ah, Al);
  k_split<<<(unsigned)(((int64_t)N * K + 255) / 256), 256, 0, s>>>(B, (int64_t)N * K, Bh, Bl);
  CUtensorMap mA2, mB2, mBh, mBl;
  if (!make_map_pair(&mA2, Ah, Al, M, K, K, BM) || !make_map_pair(&mB2, Bh, Bl, N, K, K, BN) ||
      !make_map(&mBh, Bh, N, K, K, BN) || !make_map(&mBl, Bl, N, K, K, BN))
    return BAKRON_ERR_CUDA;
  TcParams P{};
  P.mode = MODE_DENSE;
  P.K = K;
  P.row0 = 0;
  P.out_hi = C;
  P.ldo = N;
  P.status = status;
  P.spin_cycles = spin_cycles_from_env();
  dim3 grid(N / BN, M / BM);
  if (tc_pair_on() && M % (2 * BM) == 0) {
    CUtensorMap mB2h;
    if (!make_map_pair(&mB2h, Bh, Bl, N, K, K, BN_HALF)) return BAKRON_ERR_CUDA;
    BK_CUDA_OK(launch_pair(dim3(2 * (N / BN), M / (2 * BM)), s, false, mA2, mB2h, mBh, mBl, mBh,
                           mBl, P));
  } else {
    k_tc_band<V_BAND><<<grid, THREADS, SMEM_BYTES, s>>>(mA2, mB2, mBh, mBl, mBh, mBl, P);
  }
  BK_CUDA_OK(cudaGetLastError());
  return bakron_read_status(workspace, stream);
}

// ------------------------------------------------------------ Gram matrices
namespace {
constexpr int GRAM_MAX_D = 1 << 16;
}  // namespace

extern "C" size_t bakron_gram_workspace_bytes(int d, int k_chunk, int weighted) {
  if (d < 1 || d > GRAM_MAX_D || k_chunk < 1) return 0;
  const int64_t dp = round_up(d, BM), kc = round_up(k_chunk, BK);
  return 256 + (size_t)(weighted ? 4 : 2) * (size_t)dp * (size_t)kc * 4;
}

extern "C" int bakron_gram(const void* X, int xdtype, int k, int d, int64_t ldx, const float* w,
                           float alpha, float beta, float* G, int64_t ldg, void* workspace,
                           size_t workspace_bytes, int sync, void* stream) {
  if (!X || !G || !workspace || k < 1 || d < 1 || d > GRAM_MAX_D || ldx < d || ldg < d)
    return BAKRON_ERR_INVALID_ARG;
  if (xdtype != BAKRON_F32 && xdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  const int64_t dp = round_up(d, BM);
  // bf16 samples without weights: one exact bf16 plane, kind::f16 MMAs, K = 64
  // per ring slot; otherwise tf32 hi/lo planes (two, or four with weights)
  const bool bf16_ops = xdtype == BAKRON_BF16 && !w;
  const int64_t kq = bf16_ops ? 2 * BK : BK;              // chunk granularity
  const size_t per_sample = bf16_ops ? (size_t)dp * 2 : (size_t)(w ? 4 : 2) * dp * 4;
  if (workspace_bytes < 256) return BAKRON_ERR_WORKSPACE;
  int64_t kc = (int64_t)((workspace_bytes - 256) / per_sample) / kq * kq;
  kc = std::min<int64_t>(kc, round_up(k, kq));
  kc = std::min<int64_t>(kc, (int64_t)1 << 30);
  if (kc < kq) return BAKRON_ERR_WORKSPACE;
  BK_CUDA_OK(ensure_attr());
  cudaStream_t s = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  int* status = (int*)ws;
  float* Th = (float*)(ws + 256);
  float* Tl = Th + dp * kc;
  float* Wh = w ? Tl + dp * kc : nullptr;
  float* Wl = w ? Wh + dp * kc : nullptr;
  BK_CUDA_OK(cudaMemsetAsync(status, 0, 256, s));
  const int nb = (int)(dp / BM);
  const unsigned ntri = (unsigned)((int64_t)nb * (nb + 1) / 2);
  const long long spin = spin_cycles_from_env();
  for (int64_t t0 = 0; t0 < k; t0 += kc) {
    const int64_t kcl = std::min<int64_t>(kc, round_up(k - t0, kq));   // this chunk's K
    dim3 sg((unsigned)(kcl / 32), (unsigned)(dp / 32));
    CUtensorMap mA2, mB2;
    if (bf16_ops) {
      __nv_bfloat16* Tb = (__nv_bfloat16*)(ws + 256);
      const int vec_ok = ((uintptr_t)X % 16 == 0 && ldx % 8 == 0) ? 1 : 0;
      dim3 tg((unsigned)(kcl / TR_TILE), (unsigned)(dp / TR_TILE));
      k_gram_transpose_bf16<<<tg, 256, 0, s>>>((const __nv_bfloat16*)X, k, d, ldx, (int)t0,
                                               (int)kc, vec_ok, Tb);
      BK_CUDA_OK(cudaGetLastError());
      if (!make_map_bf16(&mA2, Tb, dp, kcl, kc, BM) || !make_map_bf16(&mB2, Tb, dp, kcl, kc, BN))
        return BAKRON_ERR_CUDA;
    } else {
      k_gram_split<<<sg, dim3(32, 8), 0, s>>>(X, xdtype, k, d, ldx, (int)t0, (int)kc, w, Th, Tl,
                                              Wh, Wl);
      BK_CUDA_OK(cudaGetLastError());
      const float* ah = w ? Wh : Th;
      const float* al = w ? Wl : Tl;
      if (!make_map_pair(&mA2, ah, al, dp, kcl, kc, BM) ||
          !make_map_pair(&mB2, Th, Tl, dp, kcl, kc, BN))
        return BAKRON_ERR_CUDA;
    }
    TcParams P{};
    P.mode = MODE_GRAM;
    P.K = (int)kcl;
    P.out_hi = G;
    P.ldo = ldg;
    P.status = status;
    P.spin_cycles = spin;
    P.alpha = alpha;
    P.beta = t0 == 0 ? beta : 1.f;
    P.dreal = d;
    P.b_exact = xdtype == BAKRON_BF16;              // bf16 is exact in tf32: lo plane zero
    P.a_exact = xdtype == BAKRON_BF16 && !w;
    // bf16: K counted in 128-byte rows of 64; exact products, GRAM_KGROUP
    // slots (256 samples) per accumulator hand-over
    if (bf16_ops) {
      P.K = (int)(kcl / 2);
      k_tc_band<V_GRAM_BF16><<<ntri, THREADS, SMEM_BYTES, s>>>(mA2, mB2, mB2, mB2, mB2, mB2, P);
    } else {
      k_tc_band<V_GRAM_TF32><<<ntri, THREADS, SMEM_BYTES, s>>>(mA2, mB2, mB2, mB2, mB2, mB2, P);
    }
    BK_CUDA_OK(cudaGetLastError());
  }
  if (!sync) return BAKRON_OK;
  return bakron_read_status(workspace, stream);
}

extern "C" int bakron_sample_sqnorms(const void* Y, int ydtype, int k, int d, int64_t ldy,
                                     float* out, void* stream) {
  if (!Y || !out || k < 1 || d < 1 || ldy < d) return BAKRON_ERR_INVALID_ARG;
  if (ydtype != BAKRON_F32 && ydtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  k_sqnorms<<<(unsigned)(((int64_t)k * 32 + 255) / 256), 256, 0, s>>>(Y, ydtype, k, d, ldy, out);
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}
