// bakron_solve: grid parameters, the anti-diagonal leaf wavefront and the
// bulk error propagation of Alg. 5, driven over a grid of TILE x TILE tiles.
//
// Schedule (paper, Alg. 5 applied to tiles).  Tile (I, J) lies on tile
// anti-diagonal K = I + J.  rec(k, l) over tile anti-diagonals: a single
// anti-diagonal is a leaf (all its tiles are independent: an error at (i, j)
// only reaches (p, q) with i <= p and j <= q, Appendix eq. batched-feedback);
// otherwise h = floor((k + l) / 2), rec(k, h), then the band update
//     X[S2] += Pi_{S2}( L^B E_{S1} L^A^T ),  S1 = tiles on [k, h), S2 = [h, l)
// as two restricted band products (Appendix, complexity of BaKron):
//     M[I, J'] = sum_{I'} L^B[I, I'] E[I', J']       (stage 1, band S1)
//     X[I, J] += sum_{J'} M[I, J'] L^A[J, J']^T      (stage 2, outputs in S2)
// then rec(h, l).  The equivalence proof's induction goes through with tile
// ranges as active sets because no tile on a later anti-diagonal precedes a
// tile on an earlier one.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>

#include "common.cuh"
#include "profile.cuh"
#include "tc_gemm.cuh"
#include "tune.cuh"
#include "solve.cuh"
#include <stdlib.h>

#include <type_traits>

#include <algorithm>
#include <mutex>

namespace bakron {

// ------------------------------------------------------------------ grid
// One warp per (row, group): xmin = min(0, min w), xmax = max(0, max w)
// ([-1, 1] if both are 0), s = (xmax - xmin) / qmax, z = rint(-xmin / s),
// all in IEEE fp32 so the scales equal the oracle's bit for bit.
__global__ void k_grid(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G,
                       int qmax, float* scales, float* zeros, unsigned long long* stamp) {
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  stamp_begin(stamp);
  if (warp >= (int64_t)m * G) return;
  const int row = (int)(warp / G), grp = (int)(warp % G);
  const int c0 = grp * gsz, c1 = c0 + gsz;
  float mn = INFINITY, mx = -INFINITY;
  for (int c = c0 + lane; c < c1; c += 32) {
    float v = (wdt == BAKRON_BF16)
                  ? __bfloat162float(((const __nv_bfloat16*)W)[(int64_t)row * ldw + c])
                  : ((const float*)W)[(int64_t)row * ldw + c];
    mn = fminf(mn, v);
    mx = fmaxf(mx, v);
  }
  for (int o = 16; o; o >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  if (lane == 0) {
    float xmin = fminf(mn, 0.f), xmax = fmaxf(mx, 0.f);
    if (xmin == 0.f && xmax == 0.f) { xmin = -1.f; xmax = 1.f; }
    const float s = __fdiv_rn(__fsub_rn(xmax, xmin), (float)qmax);
    scales[(int64_t)row * G + grp] = s;
    zeros[(int64_t)row * G + grp] = rintf(__fdiv_rn(-xmin, s));
  }
  stamp_end(stamp);
}

// Symmetric alphabet {-l, ..., +l} of the paper's experiments (Appendix
// "Experiments"): per (row, group) the scale starts at max |w| / l and may
// shrink by up to a factor of 2; of the K + 1 candidates
//     s_k = fl(amax * fl((2K - k) / (2K l))),  k = 0..K   (K = 0: fl(1 / l))
// the one with the least round-to-nearest squared error
//     sum_q (s_k clamp(rint(w_q / s_k), -l, l) - w_q)^2
// wins, the first on ties.  w_q / s_k is formed as w_q * fl(1 / s_k): it can
// only move a value lying within rounding of a midpoint between two levels
// to the other level, where both have the same squared error.  An all-zero row/group uses amax = 1.  Stored in
// the affine form the solve reads: z = l, codes 0..2l.  One block of
// GRID_SYM_THREADS per (row, group); the row is re-read from L1 per
// candidate; sums are fp32 per thread, then a fixed tree.
constexpr int GRID_SYM_THREADS = 256;

__device__ __forceinline__ float block_sum_or_max(float v, bool is_max, float* red) {
  for (int o = 16; o; o >>= 1) {
    const float u = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, u) : v + u;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();                       // red[] free from the last call
  if (lane == 0) red[warp] = v;
  __syncthreads();
  v = red[0];
  for (int w = 1; w < GRID_SYM_THREADS / 32; ++w) v = is_max ? fmaxf(v, red[w]) : v + red[w];
  return v;
}

__global__ void __launch_bounds__(GRID_SYM_THREADS)
    k_grid_sym(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G, int levels,
               int K, float* scales, float* zeros) {
  __shared__ float red[GRID_SYM_THREADS / 32];
  const int64_t items = (int64_t)m * G;
  // block-uniform loop: every thread of a block reaches the same barriers
  for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
    const int row = (int)(item / G), grp = (int)(item % G);
    const int64_t base = (int64_t)row * ldw + (int64_t)grp * gsz;
    auto load = [&](int c) -> float {
      return (wdt == BAKRON_BF16) ? __bfloat162float(((const __nv_bfloat16*)W)[base + c])
                                  : ((const float*)W)[base + c];
    };
    float amax = 0.f;
    for (int c = threadIdx.x; c < gsz; c += GRID_SYM_THREADS) amax = fmaxf(amax, fabsf(load(c)));
    amax = block_sum_or_max(amax, true, red);
    if (amax == 0.f) amax = 1.f;
    const float L = (float)levels;
    float best_s = 0.f, best_err = INFINITY;
    for (int k = 0; k <= K; ++k) {
      const float t = K == 0 ? __fdiv_rn(1.f, L)
                             : __fdiv_rn((float)(2 * K - k), (float)(2 * K * levels));
      const float s = __fmul_rn(amax, t), rs = __fdiv_rn(1.f, s);
      float err = 0.f;
      for (int c = threadIdx.x; c < gsz; c += GRID_SYM_THREADS) {
        const float v = load(c);
        const float q = fminf(fmaxf(rintf(v * rs), -L), L);
        const float d = fmaf(s, q, -v);
        err = fmaf(d, d, err);
      }
      err = block_sum_or_max(err, false, red);
      if (k == 0 || err < best_err) { best_err = err; best_s = s; }
    }
    if (threadIdx.x == 0) {
      scales[item] = best_s;
      zeros[item] = L;
    }
  }
}

int launch_grid_sym(const void* W, int wdt, int m, int n, int64_t ldw, int levels,
                    int group_size, int shrink_steps, float* scales, float* zeros,
                    cudaStream_t s) {
  const int gsz = group_size == 0 ? n : group_size;
  const int G = n / gsz;
  const int64_t blocks = std::min<int64_t>((int64_t)m * G, 152 * 16);
  k_grid_sym<<<(unsigned)blocks, GRID_SYM_THREADS, 0, s>>>(
      W, wdt, m, n, ldw, gsz, G, levels, shrink_steps, scales, zeros);
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}

// X <- W widened to fp32 over the padded mp x np workspace (zeros outside).
// Grid-stride over chunks of 8 entries of a row (np is a multiple of 128, so
// a chunk never straddles a row), stored as two 16-byte vectors.
__global__ void k_init(const void* W, int wdt, int m, int n, int64_t ldw, float* X,
                       int64_t mp, int64_t np, unsigned long long* stamp) {
  pdl_wait();
  pdl_trigger();
  stamp_begin(stamp);
  const int64_t chunks = mp * np / 8;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < chunks;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t idx = 8 * i, r = idx / np, c = idx - r * np;
    float v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      v[j] = 0.f;
      if (r < m && c + j < n)
        v[j] = (wdt == BAKRON_BF16)
                   ? __bfloat162float(((const __nv_bfloat16*)W)[r * ldw + c + j])
                   : ((const float*)W)[r * ldw + c + j];
    }
    float4* o = reinterpret_cast<float4*>(X + idx);
    o[0] = make_float4(v[0], v[1], v[2], v[3]);
    o[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
  stamp_end(stamp);
}

__global__ void k_copy_out(const float* X, int64_t np, int m, int n, float* out) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= (int64_t)m * n) return;
  const int64_t r = idx / n, c = idx % n;
  out[idx] = X[r * np + c];
}

// Leaf blocks of a factor buffer (FactorLayout), one thread per stored float:
// block d of tile row I of L^B is L^B[I, I-d], row-major for d = 0
// (element (p, i) at p * LD + i) and k-major for d >= 1 (at i * LD + p); block
// g of tile column J of L^A is L^A[J, J-g], k-major (element (q, j) at
// j * LD + q).  Zero outside the matrix (I - d < 0) and in columns TILE..LD-1.
__global__ void k_leaf_blocks(const float* hi, const float* lo, int64_t ld, int64_t T,
                              bool row_major_diag, float* out) {
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= T * LEAF_BLOCKS * LEAF_BLOCK_FLOATS) return;
  const int c = (int)(idx % LEAF_BLOCK_LD);
  const int r = (int)((idx / LEAF_BLOCK_LD) % TILE);
  const int d = (int)((idx / LEAF_BLOCK_FLOATS) % LEAF_BLOCKS);
  const int64_t I = idx / ((int64_t)LEAF_BLOCK_FLOATS * LEAF_BLOCKS);
  float v = 0.f;
  if (c < TILE && I - d >= 0) {
    const bool rm = row_major_diag && d == 0;
    const int p = rm ? r : c, i = rm ? c : r;   // element (p, i) of the block
    const int64_t o = (TILE * I + p) * ld + TILE * (I - d) + i;
    v = hi[o] + lo[o];
  }
  out[idx] = v;
}

int build_leaf_blocks(const FactorLayout& fl, char* f, cudaStream_t s) {
  const int64_t nb = fl.Mt * LEAF_BLOCKS * LEAF_BLOCK_FLOATS, na = fl.Nt * LEAF_BLOCKS * LEAF_BLOCK_FLOATS;
  k_leaf_blocks<<<(unsigned)((nb + 255) / 256), 256, 0, s>>>(
      (const float*)(f + fl.off_LBH), (const float*)(f + fl.off_LBL), fl.mp, fl.Mt, true,
      (float*)(f + fl.off_LBblk));
  k_leaf_blocks<<<(unsigned)((na + 255) / 256), 256, 0, s>>>(
      (const float*)(f + fl.off_LAH), (const float*)(f + fl.off_LAL), fl.np, fl.Nt, false,
      (float*)(f + fl.off_LAblk));
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}

// ------------------------------------------------------------------ leaf
// One CTA rounds one TILE x TILE tile whose inbound updates from all earlier
// tiles are already in X (paper, the parallel anti-diagonal loop of Sec. 3.3,
// run inside the tile).  Lane q of a warp stands for column q; at in-tile step
// d the entry (p, q), p = d - q, is rounded.
//
// Intra-tile feedback, with G_q[i] = sum_{j<=q} e_ij L^A[q][j] (row i's
// committed errors seen from column q), is
//     x_pq = X_pq + sum_i L^B[p][i] G_q[i].
// Errors committed on the last few steps reach (p, q) only from a few
// entries up and to the left of it, because L^B and L^A are lower triangular
// with a unit diagonal: step d - t contributes the entries (p - a, q - b)
// with a + b = t, weighted L^B[p][p-a] L^A[q][q-b].  So the work splits into
//   * the chain (warp 0, lane q = column q): adds the errors of the last two
//     or three steps explicitly (in registers and shuffles) to a partial pre
//     and rounds, step after step;
//   * three helper warps (12 rows of G each): fold older errors into G and
//     form the partial pre of later steps, sum_i L^B[p][i] G_q[i] (+ X_pq),
//     which they leave in shared memory.
// The two sides hand over once per two steps (one barrier); see the
// wavefront below for the exact lag.  A step is latency bound (a shuffle and
// about seven dependent floating-point operations), and every warp of the
// leaf issues from a scheduler of its own: errors are broadcast indexed by
// row (every row written every step, zero when off the tile), a helper keeps
// its L^A values in registers rotated by 8 every 8 steps (compile-time slots)
// and loads the L^B rows of its dot products one interval ahead, and codes
// are staged in shared memory and stored coalesced at the end.
// x / s is evaluated as the exact product x * fl(1/s), rounded once to an
// integer; fl(1/s) can differ from 1/s by half an ulp, which only matters
// within 1e-6 grid units of a rounding boundary.
// Outputs: codes, X (pre-rounding values), E^T as a tf32 hi/lo pair and in
// fp32, and the tile's final G (for the window of the tiles below it).
// Three helper warps, so that each of the SM's four schedulers runs one warp
// of the leaf (warp w issues from scheduler w mod 4) and the chain shares its
// scheduler with nobody; 12 rows each (the last one's rows 32..35 are padding
// with zero errors and zero L^B).
constexpr int LEAF_HELPERS = 3;
constexpr int LEAF_THREADS = 32 * (1 + LEAF_HELPERS);
constexpr int LEAF_ROWS_PER_HELPER = 12;
constexpr int LEAF_ROWS_PADDED = LEAF_HELPERS * LEAF_ROWS_PER_HELPER;   // 36
static_assert(LEAF_ROWS_PADDED >= TILE && LEAF_ROWS_PADDED <= 36 && LEAF_ROWS_PER_HELPER % 4 == 0,
              "helper rows: float4 groups inside the 36-wide LBs rows");
constexpr int LEAF_PER_THREAD = (TILE * TILE + LEAF_THREADS - 1) / LEAF_THREADS;

// Everything a leaf reads besides its tile coordinates.
struct LeafArgs {
  int Mt, Nt, m, n;
  float* X;
  int64_t ldx;
  float *EtH, *EtL;
  float* EtF;                  // E^T in fp32 (the leaves' own copy), same layout
  float* Gout;                 // final G of every tile, X's layout (row i, column q)
  int64_t ldt;
  const float *LBblk, *LAblk;  // the factor buffer's leaf blocks
  const float *scales, *zeros;
  int G, gsz, qmax;
  uint8_t* codes;
  int* status;
  unsigned long long* stamp;   // timeline stamp slot of the launch (null: none)
  long long* clk;              // diagnostic: the chain's clock64 around its steps (null: none)
};

constexpr int KM = 36;   // row stride of k-major product operands: float4 rows
static_assert(KM == LEAF_BLOCK_LD, "the factor buffer's leaf blocks are copied as they are");

// A leaf absorbs the errors of at most this many earlier anti-diagonals of
// its block (Alg. 5 ranges of up to LEAF_WINDOW + 1 anti-diagonals are run
// as such blocks of leaves), through the E tiles (I, J - g) and the final G
// of the tiles (I - dp, J), 1 <= g, dp <= LEAF_WINDOW.
constexpr int LEAF_WINDOW = 15;
static_assert(LEAF_WINDOW + 1 == LEAF_BLOCKS, "a window needs the blocks L[I, I-1 .. I-LEAF_WINDOW]");

// Rounding to the nearest integer (ties to even) by the shift LEAF_R =
// 1.5 * 2^23: for |v| < 2^22, fl(v + LEAF_R) - LEAF_R is v rounded to an
// integer, and the clamp to integer bounds commutes with it, so
//     c - z = clamp(fl(x * fl(1/s) + LEAF_R), LEAF_R - z, LEAF_R + qmax - z) - LEAF_R
// (one fused multiply-add: the product x * fl(1/s) is rounded once, to the
// integer).  Larger |v| fall outside the bounds and are clamped.
constexpr float LEAF_R = 12582912.f;

// 32^3 products a window-P leaf forms before its wavefront (T1 and U).
__host__ __device__ constexpr int window_products(int P) { return 2 * P; }

struct LeafSmem {
  float Xs[TILE][TILE];                   // W after inbound updates
  __align__(16) float LBs[TILE][36];      // stride 36: conflict-free float4 row reads
  __align__(16) float LA0[TILE][KM];      // LA0[j][q] = L^A[J,J][q][j]
  float T1s[TILE][TILE + 1];              // T1, the initial G of a window-P leaf (P >= 1)
  __align__(16) float Ebr[4][LEAF_ROWS_PADDED];   // errors of a step, by row (ring of 4 steps)
  float Part[4][LEAF_HELPERS][TILE];              // partial pre of a step (ring of 4 steps)
  float4 Lsub[TILE];                              // (L^B[p][p-1], L^B[p][p-2], L^B[p][p-3], 0)
  __align__(16) float4 Srzl[TILE][TILE];          // (s, 1/s, R - z, R + qmax - z) per entry
  union {
    struct {   // prologue of a window-P leaf: its window, staged one d at a time
      // buffer b holds the operands of one d: [0] E[I, J-d] k-major
      // (Et[j][i] = E[i][j]), [1] G[I-d, J] (row i, column q), [2] L^A[J, J-d]
      // k-major ([j][q] = L^A[q][j]), [3] L^B[I, I-d] k-major ([i][p] =
      // L^B[p][i]).  Buffers 0, 1 alternate before the PDL wait, 2 is d = 1.
      __align__(16) float B[3][4][TILE][KM];
    } pro;
    struct {   // the wavefront
      float EsT[TILE][TILE + 1];              // after the wavefront: E transposed
      __align__(8) float2 XE[TILE][TILE];     // (pre-rounding value, error)
      uint8_t Cs[TILE][TILE];
    } w;
  } u;
};

// C[r][c] = sum_k At[k][r] B(k, c) for the 4 x 2 block of thread t < 128
// (rows 4 (t >> 4) .. +3, columns 2 (t & 15) .. +1), k ascending.  At is
// k-major with row stride KM; B(k, c) = B[k * bsk + c * bsc].
__device__ __forceinline__ void mm_4x2(const float* At, const float* B, int bsk, int bsc, int t,
                                       float (&acc)[4][2]) {
  const int r = 4 * (t >> 4), c = 2 * (t & 15);
#pragma unroll
  for (int i = 0; i < 4; ++i) acc[i][0] = acc[i][1] = 0.f;
#pragma unroll 8
  for (int k = 0; k < TILE; ++k) {
    const float4 av = *reinterpret_cast<const float4*>(At + k * KM + r);
    const float b0 = B[k * bsk + c * bsc], b1 = B[k * bsk + (c + 1) * bsc];
    acc[0][0] = fmaf(av.x, b0, acc[0][0]);
    acc[0][1] = fmaf(av.x, b1, acc[0][1]);
    acc[1][0] = fmaf(av.y, b0, acc[1][0]);
    acc[1][1] = fmaf(av.y, b1, acc[1][1]);
    acc[2][0] = fmaf(av.z, b0, acc[2][0]);
    acc[2][1] = fmaf(av.z, b1, acc[2][1]);
    acc[3][0] = fmaf(av.w, b0, acc[3][0]);
    acc[3][1] = fmaf(av.w, b1, acc[3][1]);
  }
}

// The leaf's warps (0 .. 4) synchronise on hardware barrier 1 only, so a CTA
// with more warps can run a leaf while the others wait elsewhere.
__device__ __forceinline__ void leaf_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(LEAF_THREADS) : "memory");
}

// 16-byte asynchronous copy global -> shared (L2 only); !valid writes zeros
// and reads nothing.
__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// waits until at most N of this thread's committed groups are in flight
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Copies one leaf block (TILE rows of KM floats) as it is; thread t of the leaf.
__device__ __forceinline__ void copy_block(float* dst, const float* src, int t) {
  constexpr int CHUNKS = TILE * KM / 4;
#pragma unroll
  for (int c = t; c < CHUNKS; c += LEAF_THREADS) cp_async16(dst + 4 * c, src + 4 * c, true);
}

// How a leaf learns that its inputs are ready.
//   LEAF_PDL   one launch per anti-diagonal: programmatic dependent launch
//              (everything the previous leaf wrote is ready at pdl_wait);
//   LEAF_PLAIN inside a persistent subtree, after a grid-wide barrier;
//   LEAF_FLOW  one launch per block of anti-diagonals, persistent CTAs: a tile
//              waits only for the tiles its window reads, through per-tile
//              flags that each tile sets as soon as its fp32 errors and final
//              G are in memory (before the rest of its epilogue).
constexpr int LEAF_PDL = 0, LEAF_PLAIN = 1, LEAF_FLOW = 2;

// Per-tile readiness flags of a block launch (LEAF_FLOW).
struct FlowCtx {
  unsigned* done;        // per padded tile I * ntp + J: nonzero once published
  int ntp;
  long long spin_cycles; // bound of every wait
};

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Thread 0 waits, for at most fc.spin_cycles, until tiles (I1, J1) and
// (I2, J2) are published (a tile with a negative coordinate does not exist
// and counts as published), then the leaf's threads meet at its barrier.
// A wait that runs out records BAKRON_ERR_TIMEOUT and the leaf goes on.
__device__ __forceinline__ void flow_wait(const FlowCtx& fc, int I1, int J1, int I2, int J2,
                                          int* status) {
  if (threadIdx.x == 0) {
    const int is[2] = {I1, I2}, js[2] = {J1, J2};
    for (int u = 0; u < 2; ++u) {
      if (is[u] < 0 || js[u] < 0) continue;
      const unsigned* f = fc.done + (int64_t)is[u] * fc.ntp + js[u];
      if (ld_acquire_u32(f)) continue;
      const long long t0 = clock64();
      while (!ld_acquire_u32(f)) {
        if (clock64() - t0 > fc.spin_cycles) {
          raise_status(status, BAKRON_ERR_TIMEOUT);
          break;
        }
        __nanosleep(64);   // leave the issue slots to the wavefronts sharing the SM
      }
    }
  }
  leaf_sync();
}

// Rounds tile (I, J); run by threads 0 .. LEAF_THREADS-1 of the CTA.  With
// PDL, the factor blocks and the grid (read-only during the solve, the grid
// written by the solve's first kernel, more than one kernel ago), and the
// window's terms from tiles two or more anti-diagonals back, are handled
// before waiting for the previous kernel.
//
// A window-P leaf (1 <= P <= LEAF_WINDOW) also applies everything the P
// anti-diagonals before it in its block send to it, i.e. the Alg. 5 nodes
// inside the block: for tile (I, J) that is the sum over the E tiles
// (I - dp, J - g), 1 <= dp + g <= P, of L^B[I,I-dp] E[I-dp,J-g] L^A[J,J-g]^T.
// The terms of row I (dp = 0) enter the wavefront as the initial value of G
// (which the wavefront multiplies by L^B[I,I] anyway):
//     T1 = sum_g E[I,J-g] L^A[J,J-g]^T.
// The others are added to X before the wavefront:
//     U = sum_dp L^B[I,I-dp] N_dp,   N_dp = sum_g E[I-dp,J-g] L^A[J,J-g]^T,
// and N_dp is the final G of tile (I - dp, J), which that tile's leaf leaves
// behind (its window is P - dp).  Tiles outside the matrix are zeros.
// In LEAF_FLOW mode the window's tiles come from the same launch: the tiles
// two anti-diagonals back are waited for before the products of d >= 2, the
// two neighbours before those of d = 1, and `first` (the CTA's first tile)
// also waits for the previous kernel.
template <int MODE, int P>
__device__ __forceinline__ void leaf_tile(const LeafArgs& a, int I, int J, LeafSmem& S,
                                          const FlowCtx* fc = nullptr, bool first = false) {
  static_assert(P >= 0 && P <= LEAF_WINDOW, "window");
  constexpr bool PDL = MODE == LEAF_PDL;
  static_assert(LEAF_PER_THREAD * LEAF_THREADS == TILE * TILE, "whole tile per pass");
  const int t = threadIdx.x, w = t >> 5, lane = t & 31;
  const int64_t r0 = (int64_t)I * TILE, c0 = (int64_t)J * TILE;
  // Factor blocks and the grid (read-only during the solve; the grid written
  // by the solve's first kernel, more than one kernel ago), loaded before
  // waiting for the previous kernel; the factor blocks as asynchronous copies
  // of the factor buffer's leaf blocks, which hold them in the layouts used
  // here (LBs row-major, the others k-major, rows padded to KM).
  const float* lbk = a.LBblk + (int64_t)I * LEAF_BLOCKS * LEAF_BLOCK_FLOATS;
  const float* lak = a.LAblk + (int64_t)J * LEAF_BLOCKS * LEAF_BLOCK_FLOATS;
  copy_block(&S.LBs[0][0], lbk, t);
  copy_block(&S.LA0[0][0], lak, t);
  // The window.  N_d of this tile (the errors of row I - d of the window
  // seen from column block J) equals the final G of tile (I - d, J), which
  // sits at position P - d of the same block: every leaf leaves its final G
  // in the Gout plane.  So
  //     T1 = sum_{d=1..P} E[I, J-d] L^A[J, J-d]^T,
  //     U  = sum_{d=1..P} L^B[I, I-d] G[I-d, J],
  // 2P products of 32^3, taken one d at a time.  For d >= 2 the tiles were
  // written by kernels that had completed when this one was launched: their
  // part runs before the wait for the previous kernel (overlapping it), its
  // operands double-buffered; E[I, J-1] and G[I-1, J] come after.  Thread t
  // forms rows pr .. pr+3, columns pc, pc+1 of T1 and U.
  const int pr = 4 * (t >> 4), pc = 2 * (t & 15);
  float t1[4][2], u[4][2];
#pragma unroll
  for (int i = 0; i < 4; ++i) t1[i][0] = t1[i][1] = u[i][0] = u[i][1] = 0.f;
  auto fetch_factors = [&](int d, int b) {
    copy_block(&S.u.pro.B[b][2][0][0], lak + d * LEAF_BLOCK_FLOATS, t);
    copy_block(&S.u.pro.B[b][3][0][0], lbk + d * LEAF_BLOCK_FLOATS, t);
  };
  // E[I, J-d] (row j of the buffer is the E^T row c0 - 32 d + j, columns
  // r0 ..) and G[I-d, J] (row i is the Gout row r0 - 32 d + i, columns c0 ..);
  // zeros outside the matrix
  auto fetch_tiles = [&](int d, int b) {
    constexpr int CH = TILE * TILE / 4;   // 16-byte chunks of a tile
    static_assert(CH == 2 * LEAF_THREADS, "two chunks of every tile per thread");
    const bool ve = J - d >= 0, vg = I - d >= 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = t + LEAF_THREADS * h, j = c / (TILE / 4), i4 = 4 * (c % (TILE / 4));
      cp_async16(&S.u.pro.B[b][0][j][i4],
                 ve ? a.EtF + (c0 - (int64_t)TILE * d + j) * a.ldt + r0 + i4 : a.EtF, ve);
      cp_async16(&S.u.pro.B[b][1][j][i4],
                 vg ? a.Gout + (r0 - (int64_t)TILE * d + j) * a.ldx + c0 + i4 : a.Gout, vg);
    }
  };
  // T1 += E[I, J-d] L^A[J, J-d]^T and U += L^B[I, I-d] G[I-d, J] from buffer b
  auto products = [&](int b) {
#pragma unroll 2
    for (int k = 0; k < TILE; ++k) {
      const float4 ae = *reinterpret_cast<const float4*>(&S.u.pro.B[b][0][k][pr]);
      const float be0 = S.u.pro.B[b][2][k][pc], be1 = S.u.pro.B[b][2][k][pc + 1];
      const float4 ab = *reinterpret_cast<const float4*>(&S.u.pro.B[b][3][k][pr]);
      const float bn0 = S.u.pro.B[b][1][k][pc], bn1 = S.u.pro.B[b][1][k][pc + 1];
      const float ea[4] = {ae.x, ae.y, ae.z, ae.w}, ba[4] = {ab.x, ab.y, ab.z, ab.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        t1[i][0] = fmaf(ea[i], be0, t1[i][0]);
        t1[i][1] = fmaf(ea[i], be1, t1[i][1]);
        u[i][0] = fmaf(ba[i], bn0, u[i][0]);
        u[i][1] = fmaf(ba[i], bn1, u[i][1]);
      }
    }
  };
  if (P >= 1) fetch_factors(1, 2);
  cp_async_commit();
  float scv[LEAF_PER_THREAD], zv[LEAF_PER_THREAD];
#pragma unroll
  for (int k = 0; k < LEAF_PER_THREAD; ++k) {
    const int e = t + k * LEAF_THREADS;
    const int p = e / TILE, c = e % TILE;
    const bool real = (r0 + p) < a.m && (c0 + c) < a.n;
    const int64_t og = real ? (r0 + p) * a.G + (c0 + c) / a.gsz : 0;
    scv[k] = real ? a.scales[og] : 1.f;
    zv[k] = real ? a.zeros[og] : 0.f;
  }
  // the grid of every entry, and the error ring, before the wait
#pragma unroll
  for (int k = 0; k < LEAF_PER_THREAD; ++k) {
    const int e = t + k * LEAF_THREADS;
    // the clamp bounds of the shifted rounding (LEAF_R - z, LEAF_R + qmax - z:
    // integers below 2^24, exact in fp32)
    S.Srzl[e / TILE][e % TILE] = make_float4(scv[k], 1.f / scv[k], LEAF_R - zv[k],
                                             LEAF_R + (float)a.qmax - zv[k]);
  }
  for (int e = t; e < 4 * LEAF_ROWS_PADDED; e += LEAF_THREADS) (&S.Ebr[0][0])[e] = 0.f;
  if constexpr (MODE == LEAF_FLOW) {
    if (first) {   // X was written by the kernel before this launch
      pdl_wait();
      pdl_trigger();
    }
    if (P >= 2) flow_wait(*fc, I, J - 2, I - 2, J, a.status);
  }
  if (P >= 2) {
#pragma unroll
    for (int d = 2; d <= P && d <= 3; ++d) {
      fetch_factors(d, d & 1);
      fetch_tiles(d, d & 1);
      cp_async_commit();
    }
#pragma unroll 1
    for (int d = 2; d <= P; ++d) {
      if (d < P) cp_async_wait_group<1>();   // the copies of d + 1 may still fly
      else cp_async_wait_group<0>();
      leaf_sync();
      products(d & 1);
      if (d + 2 <= P) {
        leaf_sync();   // buffer d & 1 is read: it takes d + 2
        fetch_factors(d + 2, d & 1);
        fetch_tiles(d + 2, d & 1);
        cp_async_commit();
      }
    }
  }
  // X at this thread's product positions: rows pr .. pr+3, columns pc, pc+1.
  // Inside a block only the leaves run, each writing its own anti-diagonal's
  // tiles, so for P >= 1 this tile's X was last written by the band product
  // before the block, two or more kernels ago: it is loaded before the wait.
  float xv[4][2];
  auto load_x = [&]() {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 x2 =
          __ldcg(reinterpret_cast<const float2*>(a.X + (r0 + pr + i) * a.ldx + c0 + pc));
      xv[i][0] = x2.x;
      xv[i][1] = x2.y;
    }
  };
  if (P >= 1 || !PDL) load_x();
  if constexpr (PDL) {
    pdl_wait();
    pdl_trigger();
  } else if constexpr (MODE == LEAF_FLOW) {
    if (P >= 1) flow_wait(*fc, I, J - 1, I - 1, J, a.status);
  }
  stamp_begin(a.stamp);
  if (P == 0 && PDL) load_x();
  if (P >= 1) fetch_tiles(1, 2);
  cp_async_commit();
  cp_async_wait_group<0>();
  leaf_sync();   // factor blocks and the last window tiles in shared memory
  if (P >= 1) {
    products(2);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      S.T1s[pr + i][pc] = t1[i][0];
      S.T1s[pr + i][pc + 1] = t1[i][1];
      xv[i][0] += u[i][0];
      xv[i][1] += u[i][1];
    }
  }
  leaf_sync();   // the wavefront's arrays overlay the prologue's
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    S.Xs[pr + i][pc] = xv[i][0];
    S.Xs[pr + i][pc + 1] = xv[i][1];
  }

  if (t < TILE)
    S.Lsub[t] = make_float4(t >= 1 ? S.LBs[t][t - 1] : 0.f, t >= 2 ? S.LBs[t][t - 2] : 0.f,
                            t >= 3 ? S.LBs[t][t - 3] : 0.f, 0.f);
  leaf_sync();
  // ---------------------------------------------------------- the wavefront
  // Steps go in intervals of two (steps 2k and 2k+1) with one barrier at the
  // end of each.  In interval k the helpers fold the errors of steps 2k-2 and
  // 2k-1 (published at the barrier before it) and leave the partial pre of
  // steps 2k+2 and 2k+3, so the pre of step d covers the errors of steps up
  // to d-3 (d even) or d-4 (d odd).  The chain adds the rest itself: every
  // error of the last two (three) steps that reaches (p, q), i.e. entry
  // (p-a, q-b) for 1 <= a+b <= 2 (3), with weight L^B[p][p-a] L^A[q][q-b].
  // Its own column's errors it keeps in registers (E1..E3: steps d-1..d-3);
  // those of the columns to its left (L1_*: column q-1, L2_*: q-2, L3_3:
  // q-3, each from the step its suffix names back) arrive by shuffles, and
  // only L1_1, the left neighbour's newest error, is on the critical path.
  const int q = lane;
  if (w == 0) {
    // ------------------------------------------------ the chain
    const bool col_real = (c0 + q) < a.n;
    const int rows_real = a.m - (int)r0;     // rows p < rows_real are inside W
    // entry (p, q) is real iff 0 <= p < plim (one unsigned compare per step)
    const unsigned plim = col_real ? (unsigned)min(max(rows_real, 0), TILE) : 0u;
    const float la1 = q >= 1 ? S.LA0[q - 1][q] : 0.f;
    const float la2 = q >= 2 ? S.LA0[q - 2][q] : 0.f;
    const float la3 = q >= 3 ? S.LA0[q - 3][q] : 0.f;
    constexpr float R = LEAF_R;
    float E1 = 0.f, E2 = 0.f, E3 = 0.f;
    float L1_1 = 0.f, L1_2 = 0.f, L1_3 = 0.f, L2_2 = 0.f, L2_3 = 0.f, L3_3 = 0.f;
    // One step.  Of the explicit terms only E1 (own column, last step) and
    // L1_1 (left neighbour, last step, still in flight from its shuffle) are
    // new; the sum of the older ones is formed first so that these two enter
    // last.  The shuffles the next step needs are issued as soon as their
    // inputs exist.  Entries off the tile or outside W get a zero error (the
    // factor mk).
    auto step = [&](int d, bool odd, float pre, const float4& g, const float4& lb) {
      const int p = d - q;
      const bool on_tile = (unsigned)p < (unsigned)TILE;
      float A = fmaf(la2, L2_2, pre);
      const float A2 = fmaf(lb.y, E2, (lb.x * la1) * L1_2);
      if (odd) {
        const float o1 = fmaf(la3, L3_3, (lb.x * la2) * L2_3);
        const float o2 = fmaf(lb.y * la1, L1_3, lb.z * E3);
        A = A + (o1 + o2);
      }
      A = A + A2;
      const float nL3_3 = __shfl_up_sync(0xffffffffu, L2_2, 1);   // column q-3, this step's d-2
      const float x = fmaf(la1, L1_1, fmaf(lb.x, E1, A));
      const float nL2_2 = __shfl_up_sync(0xffffffffu, L1_1, 1);   // column q-2, step d-1
      const float tc = fminf(fmaxf(fmaf(x, g.y, R), g.z), g.w);
      const float mk = (unsigned)p < plim ? 1.f : 0.f;
      const float e = fmaf(g.x, tc - R, -x) * mk;   // s (c - z) - x, rounded once
      L1_3 = L1_2;
      L1_2 = L1_1;
      L2_3 = L2_2;
      L2_2 = nL2_2;
      L3_3 = nL3_3;
      E3 = E2;
      E2 = E1;
      E1 = e;
      L1_1 = __shfl_up_sync(0xffffffffu, e, 1);                    // column q-1, step d
      if (on_tile) {
        S.u.w.XE[p][q] = make_float2(x, e);
        S.u.w.Cs[p][q] = (uint8_t)(int)(tc - g.z);
      }
      S.Ebr[d & 3][p & (TILE - 1)] = e;    // rows off the tile get a zero
    };
    // the grid and the sub-diagonal L^B of the next interval's entries are
    // loaded one interval ahead; three intervals per loop iteration, so that
    // the three-step histories (E*, L*_*) rotate by renaming
    float4 g0 = S.Srzl[(0 - q) & (TILE - 1)][q], g1 = S.Srzl[(1 - q) & (TILE - 1)][q];
    float4 lb0 = S.Lsub[(0 - q) & (TILE - 1)], lb1 = S.Lsub[(1 - q) & (TILE - 1)];
    leaf_sync();   // the helpers' pre of steps 0 and 1
    if (a.clk != nullptr && lane == 0) a.clk[0] = clock64();
#pragma unroll 3
    for (int k = 0; k < TILE; ++k) {
      const int d0 = 2 * k, d1 = 2 * k + 1;
      const float* pa = &S.Part[d0 & 3][0][q];
      const float* pb = &S.Part[d1 & 3][0][q];
      static_assert(LEAF_HELPERS == 3, "the chain sums three partials");
      const float pre0 = (pa[0] + pa[TILE]) + pa[2 * TILE];
      const float pre1 = (pb[0] + pb[TILE]) + pb[2 * TILE];
      const float4 g0c = g0, g1c = g1, lb0c = lb0, lb1c = lb1;
      const int n0 = (d0 + 2 - q) & (TILE - 1), n1 = (d1 + 2 - q) & (TILE - 1);
      g0 = S.Srzl[n0][q];
      g1 = S.Srzl[n1][q];
      lb0 = S.Lsub[n0];
      lb1 = S.Lsub[n1];
      step(d0, false, pre0, g0c, lb0c);
      if (d1 < 2 * TILE - 1) step(d1, true, pre1, g1c, lb1c);
      leaf_sync();
    }
    if (a.clk != nullptr && lane == 0) a.clk[1] = clock64();
  } else {
    // ------------------------------------------------ helpers: rows i0..i0+11
    const int g = w - 1, i0 = LEAF_ROWS_PER_HELPER * g;
    // L^A[q][j] sits in slot (j + 2 + i0 - 8b) mod 32 during steps [8b, 8b + 8)
    // (intervals 4b .. 4b+3): the column j = s - i0 - r of row i0 + r that
    // step s = 8b + 2v - 2 (+1) brings is in slot 2v - r (+1) mod 32
    float LAr[TILE];
#pragma unroll
    for (int sl = 0; sl < TILE; ++sl) LAr[sl] = S.LA0[(sl - 2 - i0) & (TILE - 1)][q];
    float Gg[LEAF_ROWS_PER_HELPER];
#pragma unroll
    for (int r = 0; r < LEAF_ROWS_PER_HELPER; ++r)
      Gg[r] = (P >= 1 && i0 + r < TILE) ? S.T1s[i0 + r][q] : 0.f;
    // The L^B row (and, for helper 0, X) of step d's entry (row d - q), zero
    // off the tile; loaded one interval before use into one of four slots
    // (slots 2, 3 serve even intervals, 0, 1 odd ones).
    float LBv[4][LEAF_ROWS_PER_HELPER], Xv[4];
    auto fetch = [&](int d, int slot) {
      const int pn = d - q;
      const bool on_tile = pn >= 0 && pn < TILE;
      const int pr = on_tile ? pn : 0;
#pragma unroll
      for (int v = 0; v < LEAF_ROWS_PER_HELPER / 4; ++v) {
        float4 l = *reinterpret_cast<const float4*>(&S.LBs[pr][i0 + 4 * v]);
        if (!on_tile) l = make_float4(0.f, 0.f, 0.f, 0.f);
        LBv[slot][4 * v] = l.x;
        LBv[slot][4 * v + 1] = l.y;
        LBv[slot][4 * v + 2] = l.z;
        LBv[slot][4 * v + 3] = l.w;
      }
      Xv[slot] = (g == 0 && on_tile) ? S.Xs[pr][q] : 0.f;
    };
    // partial pre of step d's entry over these rows (zero off the tile)
    auto dot = [&](int d, int slot) {
      float a4[LEAF_ROWS_PER_HELPER / 4];
#pragma unroll
      for (int v = 0; v < LEAF_ROWS_PER_HELPER / 4; ++v)
        a4[v] = fmaf(LBv[slot][4 * v], Gg[4 * v],
                     fmaf(LBv[slot][4 * v + 1], Gg[4 * v + 1],
                          fmaf(LBv[slot][4 * v + 2], Gg[4 * v + 2],
                               fmaf(LBv[slot][4 * v + 3], Gg[4 * v + 3], v == 0 ? Xv[slot] : 0.f))));
      static_assert(LEAF_ROWS_PER_HELPER == 12, "three float4 groups per helper");
      S.Part[d & 3][g][q] = (a4[0] + a4[1]) + a4[2];
    };
    // fold the errors of step sidx (its row i0 + r came from column sidx - i0 - r)
    auto fold = [&](int sidx, int slot0) {
      float ev[LEAF_ROWS_PER_HELPER];
#pragma unroll
      for (int v = 0; v < LEAF_ROWS_PER_HELPER / 4; ++v) {
        const float4 e4 = *reinterpret_cast<const float4*>(&S.Ebr[sidx & 3][i0 + 4 * v]);
        ev[4 * v] = e4.x;
        ev[4 * v + 1] = e4.y;
        ev[4 * v + 2] = e4.z;
        ev[4 * v + 3] = e4.w;
      }
#pragma unroll
      for (int r = 0; r < LEAF_ROWS_PER_HELPER; ++r)
        Gg[r] = fmaf(ev[r], LAr[(slot0 - r) & (TILE - 1)], Gg[r]);
    };
    // the pre of steps 0 and 1: nothing folded yet
    fetch(0, 0);
    fetch(1, 1);
    dot(0, 0);
    dot(1, 1);
    fetch(2, 2);
    fetch(3, 3);
    leaf_sync();   // the chain's interval 0 may start
#pragma unroll 1
    for (int b = 0; b < TILE / 4; ++b) {
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const int k = 4 * b + v;
        const int cur = (v & 1) ? 0 : 2, nxt = (v & 1) ? 2 : 0;
        fetch(2 * k + 4, nxt);    // rows of the next interval, ahead of their use
        fetch(2 * k + 5, nxt + 1);
        if (k >= 1) {             // steps 2k-2 and 2k-1 were published at the last barrier
          fold(2 * k - 2, 2 * v);
          fold(2 * k - 1, 2 * v + 1);
        }
        if (2 * k + 2 < 2 * TILE - 1) dot(2 * k + 2, cur);
        if (2 * k + 3 < 2 * TILE - 1) dot(2 * k + 3, cur + 1);
        leaf_sync();
      }
      // next block: the slot of every column drops by 8, i.e. new slot s = old slot s + 8
      float tmp[TILE];
#pragma unroll
      for (int j = 0; j < TILE; ++j) tmp[j] = LAr[(j + 8) & (TILE - 1)];
#pragma unroll
      for (int j = 0; j < TILE; ++j) LAr[j] = tmp[j];
    }
    if (P < LEAF_WINDOW) {
      // the final G (the last step's errors, published at the last barrier,
      // folded too; LAr is back at its first rotation) for the tiles below
      // in this block: G[i][q] = T1[i][q] + sum_{j <= q} E[i][j] L^A[J,J][q][j]
      fold(2 * TILE - 2, 0);
#pragma unroll
      for (int r = 0; r < LEAF_ROWS_PER_HELPER; ++r)
        if (i0 + r < TILE) a.Gout[(r0 + i0 + r) * a.ldx + c0 + q] = Gg[r];
    }
  }
  leaf_sync();   // the wavefront is done: its arrays are free
  // transpose E through a padded buffer (conflict-free both ways)
  for (int e = t; e < TILE * TILE; e += LEAF_THREADS) {
    const int r = e / TILE, c = e % TILE;
    S.u.w.EsT[c][r] = S.u.w.XE[r][c].y;
  }
  leaf_sync();
  if constexpr (MODE == LEAF_FLOW) {
    // what the tiles right of and below this one read (E^T in fp32; the final
    // G the helpers stored above), then the flag, then the rest
    for (int e = t; e < TILE * TILE; e += LEAF_THREADS) {
      const int r = e / TILE, c = e % TILE;
      a.EtF[(c0 + r) * a.ldt + r0 + c] = S.u.w.EsT[r][c];
    }
    leaf_sync();
    if (t == 0) {
      __threadfence();
      atomicExch(fc->done + (int64_t)I * fc->ntp + J, 1u);
    }
  }
  bool bad = false;
  for (int e = t; e < TILE * TILE; e += LEAF_THREADS) {
    const int r = e / TILE, c = e % TILE;
    const float xr = S.u.w.XE[r][c].x;
    bad |= !isfinite(xr);
    a.X[(r0 + r) * a.ldx + c0 + c] = xr;
    if ((r0 + r) < a.m && (c0 + c) < a.n) a.codes[(r0 + r) * a.n + c0 + c] = S.u.w.Cs[r][c];
    const float ev = S.u.w.EsT[r][c];        // E^T row c0 + r, column r0 + c
    const float hi = tf32_hi(ev);
    const int64_t o = (c0 + r) * a.ldt + r0 + c;
    a.EtH[o] = hi;
    a.EtL[o] = ev - hi;
    if constexpr (MODE != LEAF_FLOW) a.EtF[o] = ev;
  }
  if (bad) raise_status(a.status, BAKRON_ERR_NONFINITE);
  leaf_sync();   // shared memory free for the next tile of this CTA
  stamp_end(a.stamp);
}

// leaf_tile<MODE, P> for a window known at run time (0 <= h <= LEAF_WINDOW)
template <int MODE, int P>
__device__ __forceinline__ void leaf_tile_window(int h, const LeafArgs& a, int I, int J, LeafSmem& S,
                                                 const FlowCtx* fc = nullptr, bool first = false) {
  if (h == P || P == LEAF_WINDOW) {
    leaf_tile<MODE, P>(a, I, J, S, fc, first);
    return;
  }
  if constexpr (P < LEAF_WINDOW) leaf_tile_window<MODE, P + 1>(h, a, I, J, S, fc, first);
}

// One CTA per tile of tile anti-diagonal K; P: the leaf's window.
template <int P>
__global__ void __launch_bounds__(LEAF_THREADS) k_leaf(int K, LeafArgs a) {
  extern __shared__ __align__(16) unsigned char leaf_smem[];
  LeafSmem& S = *reinterpret_cast<LeafSmem*>(leaf_smem);
  const int I = max(0, K - (a.Nt - 1)) + blockIdx.x;
  leaf_tile<LEAF_PDL, P>(a, I, K - I, S);
}

// The leaves of anti-diagonal K of H problems of one shape in one launch
// (blockIdx.y = problem): problem h's workspace is `slice` bytes after problem
// h - 1's, its factor buffer and outputs are its own.
constexpr int MAX_HEADS = 32;
struct LeafHeads {
  LeafArgs base;       // problem 0
  int64_t slice;       // bytes between consecutive problems' workspaces
  const float* LBblk[MAX_HEADS];
  const float* LAblk[MAX_HEADS];
  uint8_t* codes[MAX_HEADS];
  const float* scales[MAX_HEADS];
  const float* zeros[MAX_HEADS];
};

template <int P>
__global__ void __launch_bounds__(LEAF_THREADS) k_leaf_heads(int K, const __grid_constant__ LeafHeads L) {
  extern __shared__ __align__(16) unsigned char leaf_smem[];
  LeafSmem& S = *reinterpret_cast<LeafSmem*>(leaf_smem);
  const int h = blockIdx.y;
  const int64_t ds = (int64_t)h * L.slice;
  LeafArgs a = L.base;
  a.X = (float*)((char*)a.X + ds);
  a.EtH = (float*)((char*)a.EtH + ds);
  a.EtL = (float*)((char*)a.EtL + ds);
  a.EtF = (float*)((char*)a.EtF + ds);
  a.Gout = (float*)((char*)a.Gout + ds);
  a.status = (int*)((char*)a.status + ds);
  a.LBblk = L.LBblk[h];
  a.LAblk = L.LAblk[h];
  a.codes = L.codes[h];
  a.scales = L.scales[h];
  a.zeros = L.zeros[h];
  const int I = max(0, K - (a.Nt - 1)) + blockIdx.x;
  leaf_tile<LEAF_PDL, P>(a, I, K - I, S);
}

// A whole block of leaves [k, l) in one launch (LEAF_FLOW).  The block's
// tiles are numbered by anti-diagonal, then row; CTAs take them in that order
// from a counter, and a tile waits only for tiles numbered before it, which
// CTAs already running hold: the lowest unfinished tile can always proceed.
struct FlowArgs {
  LeafArgs leaf;
  FlowCtx fc;
  int k, l;
  unsigned* claim;   // this launch's tile counter (zero before the launch)
};

__global__ void __launch_bounds__(LEAF_THREADS) k_leaf_flow(const __grid_constant__ FlowArgs F) {
  extern __shared__ __align__(16) unsigned char leaf_smem[];
  LeafSmem& S = *reinterpret_cast<LeafSmem*>(leaf_smem);
  __shared__ int tile_s;
  const int Mt = F.leaf.Mt, Nt = F.leaf.Nt;
  bool first = true;
  for (;;) {
    if (threadIdx.x == 0) tile_s = (int)atomicAdd(F.claim, 1u);
    leaf_sync();
    int rem = tile_s, K = F.k, I = -1;
    leaf_sync();   // every thread has read tile_s before the next claim
    for (; K < F.l; ++K) {
      const int ilo = max(0, K - (Nt - 1)), cnt = min(K, Mt - 1) - ilo + 1;
      if (rem < cnt) {
        I = ilo + rem;
        break;
      }
      rem -= cnt;
    }
    if (I < 0) break;
    leaf_tile_window<LEAF_FLOW, 0>(K - F.k, F.leaf, I, K - I, S, &F.fc, first);
    first = false;
  }
}

// ------------------------------------------------------- band products (SIMT)
// Narrow Alg. 5 nodes on CUDA cores, 32 x 32 output tile per CTA, 256 threads,
// 4 outputs each.  Ranges come from (k, h, l) in closed form.  Every operand
// tile is an exact hi + lo pair; a K step's loads are all issued at once and
// the next step's tiles are fetched into registers while the current one is
// multiplied (the steps are few, so latency, not arithmetic, is the cost).
struct Band {
  int k, h, l, Mt, Nt;
  int row_lo;   // first 32-tile row with an output tile in [h, l)
  __host__ __device__ int jout_lo(int I) const { return max(0, h - I); }
  __host__ __device__ int jout_hi(int I) const { return min(Nt - 1, l - 1 - I); }
};

constexpr int SIMT_THREADS = 256;
constexpr int SIMT_PER = TILE * TILE / SIMT_THREADS;   // 4 elements per thread per tile

// One operand tile, element e = t + SIMT_THREADS * k of the 32 x 32 block at
// (row0, col0) of a hi/lo plane pair with leading dimension ld.
// hi and lo stay separate until the tile is stored, so nothing waits on the
// loads before the next tile product has been issued.
struct TileRegs {
  float h[SIMT_PER], l[SIMT_PER];
  __device__ void load(const float* __restrict__ hi, const float* __restrict__ lo, int64_t ld,
                       int64_t row0, int64_t col0, int t) {
#pragma unroll
    for (int k = 0; k < SIMT_PER; ++k) {
      const int e = t + SIMT_THREADS * k;
      const int64_t o = (row0 + e / TILE) * ld + col0 + e % TILE;
      h[k] = __ldcg(hi + o);   // L2: coherent within a persistent kernel
      l[k] = __ldcg(lo + o);
    }
  }
  // as stored (S[r][c] = tile[r][c]) or transposed (S[c][r] = tile[r][c])
  __device__ void store(float (*S)[TILE + 1], bool transpose, int t) const {
#pragma unroll
    for (int k = 0; k < SIMT_PER; ++k) {
      const int e = t + SIMT_THREADS * k;
      const float v = h[k] + l[k];
      if (transpose) S[e % TILE][e / TILE] = v;
      else S[e / TILE][e % TILE] = v;
    }
  }
};

// acc[u] += sum_kk A[tr][kk] B[kk][tc + u]
__device__ __forceinline__ void tile_mac(const float (*A)[TILE + 1], const float (*B)[TILE + 1],
                                         int tr, int tc, float (&acc)[4]) {
#pragma unroll 8
  for (int kk = 0; kk < TILE; ++kk) {
    const float a = A[tr][kk];
#pragma unroll
    for (int u = 0; u < 4; ++u) acc[u] = fmaf(a, B[kk][tc + u], acc[u]);
  }
}

struct BandSmem {
  float As[TILE][TILE + 1];
  float Bs[TILE][TILE + 1];
  float Ts[TILE][TILE + 1];
};

// Operands of the SIMT band products.
struct BandArgs {
  const float *LBH, *LBL;
  int64_t ldb;
  const float *EtH, *EtL;
  int64_t ldt;
  const float *LAH, *LAL;
  int64_t lda;
  float *MH, *ML;
  int64_t ldm;
  float* X;
  int64_t ldx;
  unsigned long long* stamp;   // timeline stamp slot of the launch (null: none)
};

// Unit (x, y) of stage 1: M tile (I, J') with I = row_lo + y, J' = max(0, k - I) + x.
__device__ __forceinline__ bool band1_index(const Band& bd, int x, int y, int& I, int& Jp) {
  I = bd.row_lo + y;
  const int jo_hi = bd.jout_hi(I);
  if (bd.jout_lo(I) > jo_hi) return false;
  Jp = max(0, bd.k - I) + x;
  return Jp <= min(bd.h - 1, jo_hi);
}

// Unit (x, y) of stage 2 (and of the fused form): output tile (I, J) of S2.
__device__ __forceinline__ bool band2_index(const Band& bd, int x, int y, int& I, int& J) {
  I = bd.row_lo + y;
  J = bd.jout_lo(I) + x;
  return J <= bd.jout_hi(I);
}

// Stage 1: M[I, J'] = sum_{I' in S1 column J', I' <= I} L^B[I, I'] E[I', J'].
__device__ __forceinline__ void band1_unit(const Band& bd, const BandArgs& a, int I, int Jp,
                                           BandSmem& S) {
  const int i_lo = max(0, bd.k - Jp), i_hi = min(I, bd.h - 1 - Jp);
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  // two tile pairs in flight: B[kk][col] = E[I'*T + kk][J'*T + col] = E^T[J'*T + col][I'*T + kk]
  TileRegs ra[2], rb[2];
  auto fetch = [&](int j, int Ip) {
    ra[j].load(a.LBH, a.LBL, a.ldb, (int64_t)I * TILE, (int64_t)Ip * TILE, t);
    rb[j].load(a.EtH, a.EtL, a.ldt, (int64_t)Jp * TILE, (int64_t)Ip * TILE, t);
  };
  fetch(0, i_lo);
  if (i_lo + 1 <= i_hi) fetch(1, i_lo + 1);
  for (int Ip = i_lo; Ip <= i_hi; Ip += 2) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      if (Ip + j > i_hi) break;
      ra[j].store(S.As, false, t);
      rb[j].store(S.Bs, true, t);
      __syncthreads();
      if (Ip + j + 2 <= i_hi) fetch(j, Ip + j + 2);
      tile_mac(S.As, S.Bs, tr, tc, acc);
      __syncthreads();
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int64_t o = ((int64_t)I * TILE + tr) * a.ldm + (int64_t)Jp * TILE + tc + u;
    const float hi = tf32_hi(acc[u]);
    a.MH[o] = hi;
    a.ML[o] = acc[u] - hi;
  }
}

// Stage 2: X[I, J] += sum_{J' in [max(0, k - I), min(J, h - 1)]} M[I, J'] L^A[J, J']^T.
__device__ __forceinline__ void band2_unit(const Band& bd, const BandArgs& a, int I, int J,
                                           BandSmem& S) {
  const int j_lo = max(0, bd.k - I), j_hi = min(J, bd.h - 1);
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  // two tile pairs in flight: Bs[t][c] = L^A[J*T + c][J'*T + t]
  TileRegs ra[2], rb[2];
  auto fetch = [&](int j, int Jp) {
    ra[j].load(a.MH, a.ML, a.ldm, (int64_t)I * TILE, (int64_t)Jp * TILE, t);
    rb[j].load(a.LAH, a.LAL, a.lda, (int64_t)J * TILE, (int64_t)Jp * TILE, t);
  };
  fetch(0, j_lo);
  if (j_lo + 1 <= j_hi) fetch(1, j_lo + 1);
  for (int Jp = j_lo; Jp <= j_hi; Jp += 2) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      if (Jp + j > j_hi) break;
      ra[j].store(S.As, false, t);
      rb[j].store(S.Bs, true, t);
      __syncthreads();
      if (Jp + j + 2 <= j_hi) fetch(j, Jp + j + 2);
      tile_mac(S.As, S.Bs, tr, tc, acc);
      __syncthreads();
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    float* p = a.X + ((int64_t)I * TILE + tr) * a.ldx + (int64_t)J * TILE + tc + u;
    *p = __ldcg(p) + acc[u];
  }
}

// Both stages for one output tile (I, J) of S2, forming the M tiles it needs
// in shared memory,
//     X[I, J] += sum_{J'} ( sum_{I'} L^B[I, I'] E[I', J'] ) L^A[J, J']^T,
// with the same ranges as the two stages.  Narrow nodes have few (I', J')
// pairs per output, so recomputing an M tile per output costs little and
// saves a launch (or a grid-wide barrier) and the round trip of M through
// global memory.  The pairs are walked as one flat sequence so the next
// pair's tiles are in flight while the current pair is multiplied.
__device__ __forceinline__ void fused_unit(const Band& bd, const BandArgs& a, int I, int J,
                                           BandSmem& S) {
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const int j_lo = max(0, bd.k - I), j_hi = min(J, bd.h - 1);
  auto ilo = [&](int Jp) { return max(0, bd.k - Jp); };
  auto ihi = [&](int Jp) { return min(I, bd.h - 1 - Jp); };
  TileRegs ra, rb, rl;
  int Jp = j_lo, Ip = ilo(j_lo);
  if (Jp <= j_hi) {
    ra.load(a.LBH, a.LBL, a.ldb, (int64_t)I * TILE, (int64_t)Ip * TILE, t);
    rb.load(a.EtH, a.EtL, a.ldt, (int64_t)Jp * TILE, (int64_t)Ip * TILE, t);
    rl.load(a.LAH, a.LAL, a.lda, (int64_t)J * TILE, (int64_t)Jp * TILE, t);
  }
  float m4[4] = {0.f, 0.f, 0.f, 0.f};
  while (Jp <= j_hi) {
    ra.store(S.As, false, t);
    rb.store(S.Bs, true, t);
    __syncthreads();
    // next (I', J') pair of the flat walk
    int nJp = Jp, nIp = Ip + 1;
    if (nIp > ihi(Jp)) { nJp = Jp + 1; nIp = nJp <= j_hi ? ilo(nJp) : 0; }
    const bool last_of_col = nJp != Jp;
    if (nJp <= j_hi) {
      ra.load(a.LBH, a.LBL, a.ldb, (int64_t)I * TILE, (int64_t)nIp * TILE, t);
      rb.load(a.EtH, a.EtL, a.ldt, (int64_t)nJp * TILE, (int64_t)nIp * TILE, t);
    }
    tile_mac(S.As, S.Bs, tr, tc, m4);
    __syncthreads();
    if (last_of_col) {
      // M[I, J'] complete: multiply by L^A[J, J']^T
#pragma unroll
      for (int u = 0; u < 4; ++u) S.Ts[tr][tc + u] = m4[u];
      rl.store(S.Bs, true, t);
      __syncthreads();
      if (nJp <= j_hi) rl.load(a.LAH, a.LAL, a.lda, (int64_t)J * TILE, (int64_t)nJp * TILE, t);
      tile_mac(S.Ts, S.Bs, tr, tc, acc);
      __syncthreads();
#pragma unroll
      for (int u = 0; u < 4; ++u) m4[u] = 0.f;
    }
    Jp = nJp;
    Ip = nIp;
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    float* p = a.X + ((int64_t)I * TILE + tr) * a.ldx + (int64_t)J * TILE + tc + u;
    *p = __ldcg(p) + acc[u];
  }
}

// Standalone launches: grid.y walks the rows with outputs (from row_lo),
// grid.x the span of the row.
__global__ void __launch_bounds__(SIMT_THREADS) k_band1_simt(Band bd, BandArgs a) {
  pdl_wait();
  pdl_trigger();
  stamp_begin(a.stamp);
  __shared__ BandSmem S;
  int I, Jp;
  if (band1_index(bd, blockIdx.x, blockIdx.y, I, Jp)) band1_unit(bd, a, I, Jp, S);
  stamp_end(a.stamp);
}

__global__ void __launch_bounds__(SIMT_THREADS) k_band2_simt(Band bd, BandArgs a) {
  pdl_wait();
  pdl_trigger();
  stamp_begin(a.stamp);
  __shared__ BandSmem S;
  int I, J;
  if (band2_index(bd, blockIdx.x, blockIdx.y, I, J)) band2_unit(bd, a, I, J, S);
  stamp_end(a.stamp);
}

__global__ void __launch_bounds__(SIMT_THREADS) k_band_fused_simt(Band bd, BandArgs a) {
  pdl_wait();
  pdl_trigger();
  stamp_begin(a.stamp);
  __shared__ BandSmem S;
  int I, J;
  if (band2_index(bd, blockIdx.x, blockIdx.y, I, J)) fused_unit(bd, a, I, J, S);
  stamp_end(a.stamp);
}

// ------------------------------------------------- persistent subtree
// The bottom of the recursion, rec(k, l) for a narrow range, in one
// cooperative launch: its leaves and band products run as phases in the
// order rec would enqueue them, separated by grid-wide barriers instead of
// kernel boundaries.  Each phase spreads its units (tiles of a leaf, output
// or M tiles of a band stage) over the CTAs; a CTA runs a leaf with its first
// five warps and a band unit with all eight.
enum PhaseType { PH_LEAF = 0, PH_FUSED = 1, PH_STAGE1 = 2, PH_STAGE2 = 3 };
struct Phase {
  int type, k, h, l;   // a leaf: k its anti-diagonal, h its window
};
constexpr int MAX_SUBTREE = 32;  // widest range run as one subtree (anti-diagonals)
constexpr int MAX_PHASES = 128;  // >= MAX_SUBTREE leaves + 2 phases per band node

struct SubtreeArgs {
  LeafArgs leaf;
  BandArgs band;
  unsigned* bar_count;   // grid barrier: arrivals of the current generation
  unsigned* bar_gen;     // grid barrier: generation, bumped by the last arrival
  long long spin_cycles;
  int nph;
  Phase ph[MAX_PHASES];
};

// Grid-wide barrier of a cooperative launch (every CTA resident).  Thread 0
// of each CTA publishes the CTA's writes (fence), arrives on the counter and
// waits, for at most `limit` cycles, for the last arrival to bump the
// generation.  Returns false on time-out, with BAKRON_ERR_TIMEOUT recorded;
// the caller then leaves the kernel (the other CTAs time out at their next
// barrier in turn).  Data written before the barrier is read after it with
// L2 (coherent) loads.
__device__ bool grid_sync(unsigned* count, unsigned* gen, long long limit, int* status) {
  __shared__ int ok_s;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    volatile unsigned* vgen = gen;
    const unsigned g = *vgen;
    __threadfence();
    const unsigned arrived = atomicAdd(count, 1u);
    if (arrived == gridDim.x - 1) {
      atomicExch(count, 0u);
      __threadfence();
      atomicAdd(gen, 1u);
    } else {
      const long long t0 = clock64();
      while (*vgen == g) {
        if (clock64() - t0 > limit) {
          ok = 0;
          break;
        }
      }
    }
    __threadfence();
    if (!ok) raise_status(status, BAKRON_ERR_TIMEOUT);
    ok_s = ok;
  }
  __syncthreads();
  return ok_s != 0;
}

union SubtreeSmem {
  LeafSmem leaf;
  BandSmem band;
};

__global__ void __launch_bounds__(SIMT_THREADS) k_subtree(const __grid_constant__ SubtreeArgs A) {
  extern __shared__ __align__(16) unsigned char subtree_smem[];
  SubtreeSmem& S = *reinterpret_cast<SubtreeSmem*>(subtree_smem);
  const int Mt = A.leaf.Mt, Nt = A.leaf.Nt;
  for (int ph = 0; ph < A.nph; ++ph) {
    const Phase P = A.ph[ph];
    if (P.type == PH_LEAF) {
      const int ilo = max(0, P.k - (Nt - 1)), ihi = min(P.k, Mt - 1);
      if (threadIdx.x < LEAF_THREADS)
        for (int I = ilo + (int)blockIdx.x; I <= ihi; I += gridDim.x) {
          leaf_tile_window<LEAF_PLAIN, 0>(P.h, A.leaf, I, P.k - I, S.leaf);
        }
    } else {
      const int row_lo = max(0, P.h - (Nt - 1)), row_hi = min(Mt - 1, P.l - 1);
      const Band bd{P.k, P.h, P.l, Mt, Nt, row_lo};
      const int span = P.type == PH_STAGE1 ? min(P.h, P.l - P.k) : P.l - P.h;
      const int units = row_hi >= row_lo ? span * (row_hi - row_lo + 1) : 0;
      for (int u = blockIdx.x; u < units; u += gridDim.x) {
        const int x = u % span, y = u / span;
        int I, J;
        if (P.type == PH_STAGE1) {
          if (band1_index(bd, x, y, I, J)) band1_unit(bd, A.band, I, J, S.band);
        } else if (band2_index(bd, x, y, I, J)) {
          if (P.type == PH_FUSED) fused_unit(bd, A.band, I, J, S.band);
          else band2_unit(bd, A.band, I, J, S.band);
        }
      }
    }
    if (ph + 1 < A.nph && !grid_sync(A.bar_count, A.bar_gen, A.spin_cycles, A.leaf.status))
      return;
  }
}

// ---------------------------------------------------------------- driver
// CTAs of k_subtree that fit on the current device at once (occupancy x SMs),
// queried once per device; -1 on a CUDA error.
static int subtree_capacity() {
  static std::mutex mu;
  static int cap[64];
  static bool done[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return -1;
  std::lock_guard<std::mutex> lk(mu);
  if (dev < 64 && done[dev]) return cap[dev];
  int sms = 0, per_sm = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_subtree, SIMT_THREADS,
                                                    sizeof(SubtreeSmem)) != cudaSuccess)
    return -1;
  const int c = sms * per_sm;
  if (dev < 64) {
    cap[dev] = c;
    done[dev] = true;
  }
  return c;
}

struct SolveArgs {
  int m, n, Mt, Nt, G, gsz, qmax;
  int64_t mp, np;
  float *X, *EtH, *EtL, *MH, *ML;
  const float *LAH, *LAL, *LBH, *LBL;
  const float *scales, *zeros;
  uint8_t* codes;
  int* status;
  cudaStream_t s;
  // tensor-core band products for nodes spanning >= tc_min_band tile anti-diagonals
  int tc_min_band;
  int fused_max_band;   // nodes spanning <= this many tile anti-diagonals: one fused launch
  int subtree_max;      // ranges spanning <= this many: one persistent cooperative launch
  int leaf_block;       // ranges spanning <= this many: a block of leaves (1 .. LEAF_WINDOW + 1)
  int subtree_grid;     // CTAs a cooperative launch may hold (resident at once)
  bool leaf_flow;       // a block of leaves is one dataflow launch (k_leaf_flow)
  int flow_grid;        // CTAs of k_leaf_flow resident at once
  unsigned* flow_claim; // per block (by first anti-diagonal): tile counter
  unsigned* flow_done;  // per padded tile: published flag
  int ntp;              // padded tile columns
  long long spin_cycles;
  bool tc_ready;
  bool profiling;
  TcOperands tco;
  TcMaps tcm;
  LeafArgs la;
  BandArgs ba;
  int rc;
};

// Tile products each stage of node (k, h, l) must form (tile granularity):
// stage 1 over the M tiles stage 2 needs, stage 2 over the output tiles of S2.
static void band_tile_products(const SolveArgs& a, int k, int h, int l, double& p1, double& p2) {
  p1 = p2 = 0.0;
  for (int I = 0; I < a.Mt; ++I) {
    const int jlo = max(0, h - I), jhi = min(a.Nt - 1, l - 1 - I);
    if (jlo > jhi) continue;
    for (int Jp = max(0, k - I); Jp <= min(h - 1, jhi); ++Jp)
      p1 += min(I, h - 1 - Jp) - max(0, k - Jp) + 1;
    for (int J = jlo; J <= jhi; ++J) p2 += min(J, h - 1) - max(0, k - I) + 1;
  }
}

static void note(SolveArgs& a, cudaError_t e) {
  if (e != cudaSuccess) a.rc = cuda_fail(e, __FILE__, __LINE__);
}

// Leaf of anti-diagonal K; `window`: how many anti-diagonals before it (in
// its block) it absorbs.  Flops: the in-tile feedback and the window's
// products, 2 * 32^3 each, per tile.
// k_leaf<P> for a window known at run time (0 <= window <= LEAF_WINDOW)
template <int P>
static cudaError_t launch_leaf_window(int window, dim3 grid, dim3 block, size_t sm, cudaStream_t s,
                                     int K, const LeafArgs& la) {
  if (window == P || P == LEAF_WINDOW) return launch_pdl(k_leaf<P>, grid, block, sm, s, K, la);
  if constexpr (P < LEAF_WINDOW) return launch_leaf_window<P + 1>(window, grid, block, sm, s, K, la);
  return cudaErrorInvalidValue;
}
static cudaError_t launch_leaf_window(int window, dim3 grid, dim3 block, size_t sm, cudaStream_t s,
                                      int K, const LeafArgs& la) {
  return launch_leaf_window<0>(window, grid, block, sm, s, K, la);
}

template <int P>
static cudaError_t launch_heads_window(int window, dim3 grid, dim3 block, size_t sm,
                                       cudaStream_t s, int K, const LeafHeads& lh) {
  if (window == P || P == LEAF_WINDOW) return launch_pdl(k_leaf_heads<P>, grid, block, sm, s, K, lh);
  if constexpr (P < LEAF_WINDOW)
    return launch_heads_window<P + 1>(window, grid, block, sm, s, K, lh);
  return cudaErrorInvalidValue;
}

// dynamic shared memory of k_leaf<P>, k_leaf_heads<P> .. (P up to LEAF_WINDOW)
template <int P>
static cudaError_t set_leaf_smem(int bytes) {
  cudaError_t e = cudaFuncSetAttribute(k_leaf<P>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_leaf_heads<P>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if constexpr (P < LEAF_WINDOW)
    if (e == cudaSuccess) e = set_leaf_smem<P + 1>(bytes);
  return e;
}

static void leaf(SolveArgs& a, int K, int window) {
  const int ilo = max(0, K - (a.Nt - 1)), ihi = min(K, a.Mt - 1);
  LaunchScope ls(kFamLeaf, a.s,
                 2.0 * TILE * TILE * TILE * (1 + window_products(window)) * (ihi - ilo + 1));
  const dim3 grid(ihi - ilo + 1), block(LEAF_THREADS);
  const size_t sm = sizeof(LeafSmem);
  LeafArgs la = a.la;
  la.stamp = ls.stamp();
  note(a, launch_leaf_window(window, grid, block, sm, a.s, K, la));
}

// Dynamic shared memory of the leaf and subtree kernels above the 48 KB
// default, set once per process.
static cudaError_t ensure_leaf_attrs() {
  static std::mutex mu;
  static bool done = false;
  std::lock_guard<std::mutex> lk(mu);
  if (done) return cudaSuccess;
  const int sm = (int)sizeof(LeafSmem), ss = (int)sizeof(SubtreeSmem);
  cudaError_t e = set_leaf_smem<0>(sm);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_subtree, cudaFuncAttributeMaxDynamicSharedMemorySize, ss);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_leaf_flow, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
  if (e == cudaSuccess) done = true;
  return e;
}

static void band(SolveArgs& a, int k, int h, int l) {
  double p1 = 0.0, p2 = 0.0;
  if (a.profiling) band_tile_products(a, k, h, l, p1, p2);
  const double f = 2.0 * TILE * TILE * TILE;
  if (a.tc_ready && l - k >= a.tc_min_band) {
    {
      LaunchScope ls(kFamTc1, a.s, f * p1);
      int rc = tc_band_stage(1, a.tcm, a.tco, k, h, l, a.s, ls.stamp());
      if (rc != BAKRON_OK) a.rc = rc;
    }
    {
      LaunchScope ls(kFamTc2, a.s, f * p2);
      int rc = tc_band_stage(2, a.tcm, a.tco, k, h, l, a.s, ls.stamp());
      if (rc != BAKRON_OK) a.rc = rc;
    }
    return;
  }
  // rows with outputs: some J in [max(0, h - I), min(Nt - 1, l - 1 - I)]
  const int row_lo = max(0, h - (a.Nt - 1)), row_hi = min(a.Mt - 1, l - 1);
  if (row_lo > row_hi) return;
  Band bd{k, h, l, a.Mt, a.Nt, row_lo};
  // J' span per row <= min(h, l - k); output J span <= l - h
  dim3 g1(min(h, l - k), row_hi - row_lo + 1), g2(l - h, row_hi - row_lo + 1);
  BandArgs ba = a.ba;
  if (l - k <= a.fused_max_band) {
    LaunchScope ls(kFamFused, a.s, f * (p1 + p2));
    ba.stamp = ls.stamp();
    note(a, launch_pdl(k_band_fused_simt, g2, dim3(SIMT_THREADS), 0, a.s, bd, ba));
    return;
  }
  {
    LaunchScope ls(kFamBand1, a.s, f * p1);
    ba.stamp = ls.stamp();
    note(a, launch_pdl(k_band1_simt, g1, dim3(SIMT_THREADS), 0, a.s, bd, ba));
  }
  {
    LaunchScope ls(kFamBand2, a.s, f * p2);
    ba.stamp = ls.stamp();
    note(a, launch_pdl(k_band2_simt, g2, dim3(SIMT_THREADS), 0, a.s, bd, ba));
  }
}

// Phases of rec(k, l) in the order rec enqueues them.
static void subtree_phases(const SolveArgs& a, int k, int l, SubtreeArgs& A) {
  if (l - k <= a.leaf_block) {   // a block of leaves, each absorbing the ones before it
    for (int K = k; K < l; ++K) A.ph[A.nph++] = Phase{PH_LEAF, K, K - k, K + 1};
    return;
  }
  const int h = (k + l) / 2;
  subtree_phases(a, k, h, A);
  if (l - k <= a.fused_max_band) {
    A.ph[A.nph++] = Phase{PH_FUSED, k, h, l};
  } else {
    A.ph[A.nph++] = Phase{PH_STAGE1, k, h, l};
    A.ph[A.nph++] = Phase{PH_STAGE2, k, h, l};
  }
  subtree_phases(a, h, l, A);
}

static void subtree(SolveArgs& a, int k, int l) {
  SubtreeArgs A;
  A.leaf = a.la;
  A.band = a.ba;
  char* st = (char*)a.status;
  A.bar_count = (unsigned*)(st + 64);
  A.bar_gen = (unsigned*)(st + 128);
  A.spin_cycles = a.spin_cycles;
  A.nph = 0;
  subtree_phases(a, k, l, A);
  // as many CTAs as the widest leaf of the range has tiles (band phases
  // spread their units over the same CTAs)
  int widest = 1;
  for (int K = k; K < l; ++K)
    widest = max(widest, min(K, a.Mt - 1) - max(0, K - (a.Nt - 1)) + 1);
  const int grid = min(widest, a.subtree_grid);
  double flops = 0.0;
  if (a.profiling) {
    for (int i = 0; i < A.nph; ++i) {
      const Phase& P = A.ph[i];
      if (P.type == PH_LEAF) {
        flops += 2.0 * TILE * TILE * TILE * (1 + window_products(P.h)) *
                 (min(P.k, a.Mt - 1) - max(0, P.k - (a.Nt - 1)) + 1);
      } else if (P.type != PH_STAGE2) {
        double p1, p2;
        band_tile_products(a, P.k, P.h, P.l, p1, p2);
        flops += 2.0 * TILE * TILE * TILE * (p1 + p2);
      }
    }
  }
  LaunchScope ls(kFamSubtree, a.s, flops);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(SIMT_THREADS);
  cfg.dynamicSmemBytes = sizeof(SubtreeSmem);
  cfg.stream = a.s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  note(a, cudaLaunchKernelEx(&cfg, k_subtree, A));
}

// CTAs of k_leaf_flow resident at once on the current device (occupancy x
// SMs), queried once per device; -1 on a CUDA error.
static int flow_capacity() {
  static std::mutex mu;
  static int cap[64];
  static bool done[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return -1;
  std::lock_guard<std::mutex> lk(mu);
  if (dev < 64 && done[dev]) return cap[dev];
  int sms = 0, per_sm = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_leaf_flow, LEAF_THREADS,
                                                    sizeof(LeafSmem)) != cudaSuccess)
    return -1;
  const int c = sms * (per_sm > 0 ? per_sm : 1);
  if (dev < 64) {
    cap[dev] = c;
    done[dev] = true;
  }
  return c;
}

// The leaves of anti-diagonals [k, l) as one dataflow launch.
static void leaf_block_flow(SolveArgs& a, int k, int l) {
  int tiles = 0;
  double flops = 0.0;
  for (int K = k; K < l; ++K) {
    const int cnt = min(K, a.Mt - 1) - max(0, K - (a.Nt - 1)) + 1;
    tiles += cnt;
    flops += 2.0 * TILE * TILE * TILE * (1 + window_products(K - k)) * cnt;
  }
  if (tiles <= 0) return;
  LaunchScope ls(kFamLeaf, a.s, flops);
  FlowArgs F;
  F.leaf = a.la;
  F.leaf.stamp = ls.stamp();
  F.fc = FlowCtx{a.flow_done, a.ntp, a.spin_cycles};
  F.k = k;
  F.l = l;
  F.claim = a.flow_claim + k;
  note(a, launch_pdl(k_leaf_flow, dim3(min(tiles, a.flow_grid)), dim3(LEAF_THREADS),
                     sizeof(LeafSmem), a.s, F));
}

static void rec(SolveArgs& a, int k, int l) {
  if (l - k <= a.leaf_block && a.leaf_flow) {
    leaf_block_flow(a, k, l);
    return;
  }
  if (l - k <= a.leaf_block) {
    // a block of leaves: leaf K applies what anti-diagonals k .. K-1 send it
    // (the Alg. 5 nodes inside [k, l)), so no band launch is needed here
    for (int K = k; K < l; ++K) leaf(a, K, K - k);
    return;
  }
  if (l - k <= a.subtree_max && a.subtree_grid > 0) {
    subtree(a, k, l);
    return;
  }
  const int h = (k + l) / 2;
  rec(a, k, h);
  band(a, k, h, l);
  rec(a, h, l);
}

void launch_grid(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G, int qmax,
                 float* scales, float* zeros, cudaStream_t s);
int launch_init(const void* W, int wdt, int m, int n, int64_t ldw, float* X, int64_t mp,
                int64_t np, cudaStream_t s);
int launch_copy_out(const float* X, int64_t np, int m, int n, float* out, cudaStream_t s);

// Diagnostic only (bakron_diag_leaf_chain): where the leaves of the next
// solve record the chain's clock64 before and after its steps.
long long* g_diag_leaf_clk = nullptr;

// `force`: thresholds to use instead of tuning_for(m, n) (the autotuner's candidates).
// `grid_given`: scales and zeros hold the caller's grid (read only); otherwise
// the min-max grid over qmax + 1 codes is computed into them first.
// `keep_status`: leave the status word as it is (a batch of solves sharing the
// workspace keeps the first error of any of them); the grid-barrier words
// after it are cleared either way.
// The arguments of one solve of W (m x n) in `workspace` on stream s, with
// schedule tu; the tensor maps of the band stages built when they are used.
static int init_solve_args(SolveArgs& a, int m, int n, const void* factors, int qmax,
                           int group_size, uint8_t* codes, float* scales, float* zeros,
                           void* workspace, cudaStream_t s, const Tuning& tu) {
  FactorLayout fl(m, n);
  SolveLayout sl(m, n);
  char* ws = (char*)workspace;
  const char* f = (const char*)factors;
  a.m = m; a.n = n;
  a.Mt = ceil_div(m, TILE); a.Nt = ceil_div(n, TILE);
  a.gsz = group_size == 0 ? n : group_size;
  a.G = n / a.gsz;
  a.qmax = qmax;
  a.mp = sl.mp; a.np = sl.np;
  a.X = (float*)(ws + sl.off_X);
  a.EtH = (float*)(ws + sl.off_EtH);
  a.EtL = (float*)(ws + sl.off_EtL);
  a.MH = (float*)(ws + sl.off_MH);
  a.ML = (float*)(ws + sl.off_ML);
  a.LBH = (const float*)(f + fl.off_LBH);
  a.LBL = (const float*)(f + fl.off_LBL);
  a.LAH = (const float*)(f + fl.off_LAH);
  a.LAL = (const float*)(f + fl.off_LAL);
  a.scales = scales; a.zeros = zeros; a.codes = codes;
  a.status = (int*)(ws + sl.off_status);
  a.s = s;
  a.rc = BAKRON_OK;
  // the leaves' fp32 E^T and final G share the M planes (see SolveLayout)
  a.la = LeafArgs{a.Mt, a.Nt, m, n, a.X, a.np, a.EtH, a.EtL, a.MH, a.ML, a.mp,
                  (const float*)(f + fl.off_LBblk), (const float*)(f + fl.off_LAblk),
                  scales, zeros, a.G, a.gsz, a.qmax, codes, a.status, nullptr,
                  g_diag_leaf_clk};
  a.ba = BandArgs{a.LBH, a.LBL, a.mp, a.EtH, a.EtL, a.mp, a.LAH, a.LAL, a.np,
                  a.MH, a.ML, a.np, a.X, a.np, nullptr};
  a.profiling = profiling_on();
  BK_CUDA_OK(ensure_leaf_attrs());
  a.tc_min_band = tu.tc_min_band;         // 0 or less: tensor cores off
  a.fused_max_band = tu.fused_max_band;
  a.subtree_max = tu.subtree_max;         // 0 or 1: no persistent subtrees
  a.leaf_block = std::min(std::max(tu.leaf_block, 1), LEAF_WINDOW + 1);
  if (a.subtree_max > MAX_SUBTREE) a.subtree_max = MAX_SUBTREE;
  a.subtree_grid = 0;
  if (a.subtree_max >= 2) {
    const int cap = subtree_capacity();
    if (cap < 0) return BAKRON_ERR_CUDA;
    a.subtree_grid = cap;
  }
  a.spin_cycles = spin_cycles_from_env();
  a.leaf_flow = tu.leaf_flow != 0;
  a.flow_grid = 0;
  a.flow_claim = (unsigned*)(ws + sl.off_flow);
  a.flow_done = a.flow_claim + FLOW_COUNTERS;
  a.ntp = (int)(sl.np / TILE);
  if (a.leaf_flow) {
    a.flow_grid = flow_capacity();
    if (a.flow_grid <= 0) return BAKRON_ERR_CUDA;
  }
  a.tc_ready = false;
  if (a.tc_min_band > 0) {
    a.tco = TcOperands{a.mp, a.np, a.Mt, a.Nt, a.LBH, a.LBL, a.LAH, a.LAL,
                       a.EtH, a.EtL, a.MH, a.ML, a.X, a.status};
    a.tc_ready = tc_band_maps(a.tcm, a.tco);
    if (!a.tc_ready) return BAKRON_ERR_CUDA;
  }
  return BAKRON_OK;
}

int solve_impl(const void* W, int wdt, int m, int n, int64_t ldw, const void* factors, int qmax,
               int group_size, uint8_t* codes, float* scales, float* zeros, float* prerounding,
               void* workspace, cudaStream_t s, const Tuning* force, bool grid_given,
               bool keep_status) {
  SolveLayout sl(m, n);
  char* ws = (char*)workspace;
  SolveArgs a;
  {
    const Tuning tu = force ? *force : tuning_for(m, n);
    const int rc = init_solve_args(a, m, n, factors, qmax, group_size, codes, scales, zeros,
                                   workspace, s, tu);
    if (rc != BAKRON_OK) return rc;
  }
  reset_launch_count();
  if (keep_status)
    BK_CUDA_OK(cudaMemsetAsync(ws + sl.off_status + 64, 0, 256 - 64, s));
  else
    BK_CUDA_OK(cudaMemsetAsync(ws + sl.off_status, 0, 256, s));
  if (a.leaf_flow) BK_CUDA_OK(cudaMemsetAsync(ws + sl.off_flow, 0, sl.flow_bytes, s));
  if (!grid_given) launch_grid(W, wdt, m, n, ldw, a.gsz, a.G, a.qmax, scales, zeros, s);
  {
    const int rc = launch_init(W, wdt, m, n, ldw, a.X, a.mp, a.np, s);
    if (rc != BAKRON_OK) a.rc = rc;
  }
  rec(a, 0, a.Mt + a.Nt - 1);
  if (prerounding) {
    const int rc = launch_copy_out(a.X, a.np, m, n, prerounding, s);
    if (rc != BAKRON_OK) a.rc = rc;
  }
  BK_CUDA_OK(cudaGetLastError());
  return a.rc;
}

// ------------------------------------------------- problems side by side
namespace {
struct HeadsRun {
  int H;
  SolveArgs* a;               // per problem, each on its own lane
  cudaStream_t main;
  const cudaStream_t* lanes;
  cudaEvent_t fork;
  const cudaEvent_t* done;
  LeafHeads lh;
  bool on_main;               // the lanes have joined into main since the last fork
  int rc;
};

void heads_join(HeadsRun& r) {
  if (r.on_main) return;
  for (int h = 0; h < r.H; ++h) {
    if (cudaEventRecord(r.done[h], r.lanes[h]) != cudaSuccess ||
        cudaStreamWaitEvent(r.main, r.done[h], 0) != cudaSuccess)
      r.rc = BAKRON_ERR_CUDA;
  }
  r.on_main = true;
}

void heads_fork(HeadsRun& r) {
  if (!r.on_main) return;
  if (cudaEventRecord(r.fork, r.main) != cudaSuccess) r.rc = BAKRON_ERR_CUDA;
  for (int h = 0; h < r.H; ++h)
    if (cudaStreamWaitEvent(r.lanes[h], r.fork, 0) != cudaSuccess) r.rc = BAKRON_ERR_CUDA;
  r.on_main = false;
}

void heads_rec(HeadsRun& r, int k, int l) {
  const SolveArgs& a0 = r.a[0];
  if (l - k <= a0.leaf_block) {
    heads_join(r);
    for (int K = k; K < l; ++K) {
      const int ilo = max(0, K - (a0.Nt - 1)), ihi = min(K, a0.Mt - 1);
      LaunchScope ls(kFamLeaf, r.main, 2.0 * TILE * TILE * TILE * (1 + window_products(K - k)) *
                                           (ihi - ilo + 1) * r.H);
      LeafHeads lh = r.lh;
      lh.base.stamp = ls.stamp();
      const cudaError_t e = launch_heads_window<0>(K - k, dim3(ihi - ilo + 1, r.H),
                                                   dim3(LEAF_THREADS), sizeof(LeafSmem), r.main,
                                                   K, lh);
      if (e != cudaSuccess) r.rc = cuda_fail(e, __FILE__, __LINE__);
    }
    return;
  }
  const int h = (k + l) / 2;
  heads_rec(r, k, h);
  if (a0.tc_ready && l - k >= a0.tc_min_band) {
    // both stages for every problem in one tensor-core launch each, on main
    heads_join(r);
    const TcMaps* maps[MAX_HEADS];
    int* status[MAX_HEADS];
    for (int p = 0; p < r.H; ++p) {
      maps[p] = &r.a[p].tcm;
      status[p] = r.a[p].status;
    }
    double p1 = 0.0, p2 = 0.0;
    if (a0.profiling) band_tile_products(a0, k, h, l, p1, p2);
    const double f = 2.0 * TILE * TILE * TILE * r.H;
    for (int stage = 1; stage <= 2; ++stage) {
      LaunchScope ls(stage == 1 ? kFamTc1 : kFamTc2, r.main, f * (stage == 1 ? p1 : p2));
      const int rc = tc_band_stage_heads(stage, r.H, maps, status, a0.tco, k, h, l, r.main,
                                         ls.stamp());
      if (rc != BAKRON_OK) r.rc = rc;
    }
  } else {
    heads_fork(r);
    for (int p = 0; p < r.H; ++p) {
      band(r.a[p], k, h, l);
      if (r.a[p].rc != BAKRON_OK) r.rc = r.a[p].rc;
    }
  }
  heads_rec(r, h, l);
}
}  // namespace

int solve_heads_impl(int H, const void* const* W, int wdt, int m, int n, int64_t ldw,
                     const void* const* factors, int qmax, int group_size,
                     uint8_t* const* codes, float* const* scales, float* const* zeros,
                     char* workspace, size_t slice, cudaStream_t main,
                     const cudaStream_t* lanes, cudaEvent_t fork, const cudaEvent_t* done) {
  if (H < 1 || H > MAX_HEADS) return BAKRON_ERR_INVALID_ARG;
  const Tuning tu = tuning_for(m, n);
  if (tu.leaf_flow || tu.subtree_max >= 2) return BAKRON_ERR_INVALID_ARG;   // not in this schedule
  SolveLayout sl(m, n);
  SolveArgs a[MAX_HEADS];
  for (int h = 0; h < H; ++h) {
    const int rc = init_solve_args(a[h], m, n, factors[h], qmax, group_size, codes[h], scales[h],
                                   zeros[h], workspace + (size_t)h * slice, lanes[h], tu);
    if (rc != BAKRON_OK) return rc;
  }
  HeadsRun r;
  r.H = H;
  r.a = a;
  r.main = main;
  r.lanes = lanes;
  r.fork = fork;
  r.done = done;
  r.on_main = false;          // the caller forked the lanes from main
  r.rc = BAKRON_OK;
  r.lh.base = a[0].la;
  r.lh.slice = (int64_t)slice;
  for (int h = 0; h < H; ++h) {
    r.lh.LBblk[h] = a[h].la.LBblk;
    r.lh.LAblk[h] = a[h].la.LAblk;
    r.lh.codes[h] = codes[h];
    r.lh.scales[h] = scales[h];
    r.lh.zeros[h] = zeros[h];
  }
  reset_launch_count();
  // per problem on its lane: the grid-barrier words (the caller cleared the
  // status word), the grid, X from W
  for (int h = 0; h < H; ++h) {
    char* ws = workspace + (size_t)h * slice;
    BK_CUDA_OK(cudaMemsetAsync(ws + sl.off_status + 64, 0, 256 - 64, lanes[h]));
    launch_grid(W[h], wdt, m, n, ldw, a[h].gsz, a[h].G, a[h].qmax, scales[h], zeros[h], lanes[h]);
    const int rc = launch_init(W[h], wdt, m, n, ldw, a[h].X, a[h].mp, a[h].np, lanes[h]);
    if (rc != BAKRON_OK) r.rc = rc;
  }
  heads_rec(r, 0, a[0].Mt + a[0].Nt - 1);
  heads_fork(r);              // the caller joins the lanes into main at the end
  BK_CUDA_OK(cudaGetLastError());
  return r.rc;
}

// The first kernels of a solve: the min-max grid (k_grid) and X from W (k_init).
void launch_grid(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G, int qmax,
                 float* scales, float* zeros, cudaStream_t s) {
  const int64_t warps = (int64_t)m * G;
  LaunchScope ls(kFamInit, s);
  k_grid<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, s>>>(W, wdt, m, n, ldw, gsz, G, qmax,
                                                               scales, zeros, ls.stamp());
}

int launch_init(const void* W, int wdt, int m, int n, int64_t ldw, float* X, int64_t mp,
                int64_t np, cudaStream_t s) {
  const int64_t chunks = mp * np / 8;
  LaunchScope ls(kFamInit, s);
  const unsigned blocks = (unsigned)std::min<int64_t>((chunks + 255) / 256, 152 * 8);
  return BK_CUDA_RC(launch_pdl(k_init, dim3(blocks), dim3(256), 0, s, W, wdt, m, n, ldw, X, mp,
                               np, ls.stamp()));
}

int launch_solve_prologue(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G,
                          int qmax, float* scales, float* zeros, float* X, int64_t mp, int64_t np,
                          char* status_area, cudaStream_t s) {
  BK_CUDA_OK(cudaMemsetAsync(status_area, 0, 256, s));
  launch_grid(W, wdt, m, n, ldw, gsz, G, qmax, scales, zeros, s);
  return launch_init(W, wdt, m, n, ldw, X, mp, np, s);
}

int launch_copy_out(const float* X, int64_t np, int m, int n, float* out, cudaStream_t s) {
  const int64_t tot = (int64_t)m * n;
  LaunchScope ls(kFamCopy, s);
  return BK_CUDA_RC(launch_pdl(k_copy_out, dim3((unsigned)((tot + 255) / 256)), dim3(256), 0, s,
                               X, np, m, n, out));
}

}  // namespace bakron
