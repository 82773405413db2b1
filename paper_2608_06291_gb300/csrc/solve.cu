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
#include <stdlib.h>

namespace bakron {

// ------------------------------------------------------------------ grid
// One warp per (row, group): xmin = min(0, min w), xmax = max(0, max w)
// ([-1, 1] if both are 0), s = (xmax - xmin) / qmax, z = rint(-xmin / s),
// all in IEEE fp32 so the scales equal the oracle's bit for bit.
__global__ void k_grid(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G,
                       int qmax, float* scales, float* zeros) {
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
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
}

// X <- W widened to fp32 over the padded mp x np workspace (zeros outside).
__global__ void k_init(const void* W, int wdt, int m, int n, int64_t ldw, float* X,
                       int64_t mp, int64_t np) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= mp * np) return;
  const int64_t r = idx / np, c = idx % np;
  float v = 0.f;
  if (r < m && c < n)
    v = (wdt == BAKRON_BF16) ? __bfloat162float(((const __nv_bfloat16*)W)[r * ldw + c])
                             : ((const float*)W)[r * ldw + c];
  X[idx] = v;
}

__global__ void k_copy_out(const float* X, int64_t np, int m, int n, float* out) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= (int64_t)m * n) return;
  const int64_t r = idx / n, c = idx % n;
  out[idx] = X[r * np + c];
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
// Errors committed on step d - 1 reach (p, q) only through its upper
// neighbour (p - 1, q) and its left neighbour (p, q - 1), because L^B and L^A
// are lower triangular with a unit diagonal, so
//     x_pq = pre_pq + L^B[p][p-1] e_{p-1,q} + L^A[q][q-1] e_{p,q-1},
//     pre_pq = X_pq + sum_i L^B[p][i] G_q^{(d-2)}[i].
// Warp 0 runs only that two-term chain and the rounding.  Warps 1..4 each
// hold 8 rows of G for every column, fold in the errors of step d - 1 and
// leave partial sums of step d + 1's pre in shared memory, one step ahead of
// warp 0; one barrier per step orders both directions.
// A step is latency bound (about fifteen dependent floating-point operations,
// one shared-memory round and the barrier), so each step moves as few
// shared-memory words as possible: errors are broadcast indexed by row (every
// row written every step, zero when off the tile), a helper keeps its L^A
// values in registers rotated by 8 every 8 steps (compile-time slots), the
// grid and the sub-diagonal of L^B travel as one float4, and codes are staged
// in shared memory and stored coalesced at the end.
// x / s is evaluated as x * fl(1/s); it can differ from the correctly rounded
// quotient by one ulp, which only matters within 1e-6 grid units of a
// rounding boundary.
// Outputs: codes, X (pre-rounding values) and E^T as a tf32 hi/lo pair.
constexpr int LEAF_HELPERS = 4;
constexpr int LEAF_THREADS = 32 * (1 + LEAF_HELPERS);
constexpr int LEAF_ROWS_PER_HELPER = TILE / LEAF_HELPERS;
constexpr int LEAF_PER_THREAD = (TILE * TILE + LEAF_THREADS - 1) / LEAF_THREADS;

__global__ void __launch_bounds__(LEAF_THREADS)
k_leaf(int K, int Mt, int Nt, int m, int n, float* __restrict__ X, int64_t ldx,
       float* __restrict__ EtH, float* __restrict__ EtL, int64_t ldt,
       const float* __restrict__ LBH, const float* __restrict__ LBL, int64_t ldb,
       const float* __restrict__ LAH, const float* __restrict__ LAL, int64_t lda,
       const float* __restrict__ scales, const float* __restrict__ zeros, int G, int gsz,
       int qmax, uint8_t* __restrict__ codes, int* status) {
  const int I = max(0, K - (Nt - 1)) + blockIdx.x;
  const int J = K - I;
  const int t = threadIdx.x, w = t >> 5, lane = t & 31;
  __shared__ float Xs[TILE][TILE];               // W after inbound updates
  __shared__ __align__(16) float LBs[TILE][36];  // stride 36: conflict-free float4 row reads
  __shared__ float LAs[TILE][TILE + 1];
  __shared__ __align__(16) float4 Srzl[TILE][TILE];   // (s, 1/s, z, L^B[p][p-1]) per entry
  __shared__ __align__(8) float2 XE[TILE][TILE];      // (pre-rounding value, error)
  __shared__ float EsT[TILE][TILE + 1];
  __shared__ uint8_t Cs[TILE][TILE];
  __shared__ __align__(16) float Ebr[2][TILE];        // errors of a step, indexed by row
  __shared__ float Part[2][LEAF_HELPERS][TILE];
  const int64_t r0 = (int64_t)I * TILE, c0 = (int64_t)J * TILE;
  // factor blocks and grid: read-only during the solve (the grid is written by
  // the solve's first kernel, more than one kernel ago), so load before waiting
  float lbv[LEAF_PER_THREAD], lav[LEAF_PER_THREAD], scv[LEAF_PER_THREAD], zv[LEAF_PER_THREAD];
#pragma unroll
  for (int k = 0; k < LEAF_PER_THREAD; ++k) {
    const int e = t + k * LEAF_THREADS;
    if (e < TILE * TILE) {
      const int p = e / TILE, c = e % TILE;
      const int64_t ob = (r0 + p) * ldb + r0 + c, oa = (c0 + p) * lda + c0 + c;
      lbv[k] = LBH[ob] + LBL[ob];
      lav[k] = LAH[oa] + LAL[oa];
      const bool real = (r0 + p) < m && (c0 + c) < n;
      const int64_t og = (r0 + p) * G + (c0 + c) / gsz;
      scv[k] = real ? scales[og] : 1.f;
      zv[k] = real ? zeros[og] : 0.f;
    }
  }
#pragma unroll
  for (int k = 0; k < LEAF_PER_THREAD; ++k) {
    const int e = t + k * LEAF_THREADS;
    if (e < TILE * TILE) {
      const int p = e / TILE, c = e % TILE;
      LBs[p][c] = lbv[k];
      LAs[p][c] = lav[k];
    }
  }
  pdl_wait();
  pdl_trigger();
  float xv[LEAF_PER_THREAD];
#pragma unroll
  for (int k = 0; k < LEAF_PER_THREAD; ++k) {
    const int e = t + k * LEAF_THREADS;
    if (e < TILE * TILE) xv[k] = X[(r0 + e / TILE) * ldx + c0 + e % TILE];
  }
  __syncthreads();   // LBs complete: the sub-diagonal can be read
#pragma unroll
  for (int k = 0; k < LEAF_PER_THREAD; ++k) {
    const int e = t + k * LEAF_THREADS;
    if (e < TILE * TILE) {
      const int p = e / TILE, c = e % TILE;
      Xs[p][c] = xv[k];
      Srzl[p][c] = make_float4(scv[k], 1.f / scv[k], zv[k], p > 0 ? LBs[p][p - 1] : 0.f);
    }
  }
  if (t < 2 * TILE) (&Ebr[0][0])[t] = 0.f;
  for (int e = t; e < 2 * LEAF_HELPERS * TILE; e += LEAF_THREADS) (&Part[0][0][0])[e] = 0.f;
  // the pre of step 0 (row 0, only lane 0 is on the tile) is just X[0][q]; thread
  // t < 32 zeroed exactly this word above and holds X[0][t] in xv[0]
  if (t < TILE) Part[0][0][t] = xv[0];
  __syncthreads();
  const int q = lane;
  if (w == 0) {
    // ------------------------------------------------ the chain
    const bool col_real = (c0 + q) < n;
    const float la_sub = q > 0 ? LAs[q][q - 1] : 0.f;
    const float fq = (float)qmax;
    bool bad = false;
    float e_prev = 0.f;
#pragma unroll 1
    for (int d = 0; d < 2 * TILE - 1; ++d) {
      const int p = d - q;
      const bool act = p >= 0 && p < TILE;
      const int pr = p & (TILE - 1);         // the row this lane writes in Ebr
      const float e_left = __shfl_up_sync(0xffffffffu, e_prev, 1);
      float e = 0.f;
      if (act) {
        const float* part = &Part[d & 1][0][q];
        const float pre = (part[0] + part[TILE]) + (part[2 * TILE] + part[3 * TILE]);
        const float4 g = Srzl[p][q];
        const float x = fmaf(g.w, e_prev, fmaf(la_sub, e_left, pre));
        float c = rintf(x * g.y) + g.z;
        c = fminf(fmaxf(c, 0.f), fq);
        const float v = __fmul_rn(g.x, __fsub_rn(c, g.z));
        e = __fsub_rn(v, x);
        const bool real = (r0 + p) < m && col_real;
        if (!real) e = 0.f;
        bad |= !isfinite(x);
        XE[p][q] = make_float2(x, e);
        Cs[p][q] = (uint8_t)c;
      }
      Ebr[d & 1][pr] = e;
      e_prev = e;
      __syncthreads();
    }
    if (bad) raise_status(status, BAKRON_ERR_NONFINITE);
  } else {
    // ------------------------------------------------ helpers: rows i0..i0+7
    const int g = w - 1, i0 = LEAF_ROWS_PER_HELPER * g;
    // L^A[q][j] in slot (j + 1 + i0 - 8b) mod 32 during steps [8b, 8b + 8), so the
    // column j = d - 1 - i0 - r folded into row i0 + r sits in slot (u - r) mod 32
    float LAr[TILE];
#pragma unroll
    for (int s = 0; s < TILE; ++s) LAr[s] = LAs[q][(s - 1 - i0) & (TILE - 1)];
    float Gg[LEAF_ROWS_PER_HELPER];
#pragma unroll
    for (int r = 0; r < LEAF_ROWS_PER_HELPER; ++r) Gg[r] = 0.f;
#pragma unroll 1
    for (int b = 0; b < (2 * TILE) / 8; ++b) {
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int d = 8 * b + u;
        if (d < 2 * TILE - 1) {
          // fold step d-1's errors: row i0 + r came from column j = d - 1 - i0 - r
          if (d >= 1) {
            const float4 e0 = *reinterpret_cast<const float4*>(&Ebr[(d - 1) & 1][i0]);
            const float4 e1 = *reinterpret_cast<const float4*>(&Ebr[(d - 1) & 1][i0 + 4]);
            const float ev[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
#pragma unroll
            for (int r = 0; r < LEAF_ROWS_PER_HELPER; ++r)
              Gg[r] = fmaf(ev[r], LAr[(u - r) & (TILE - 1)], Gg[r]);
          }
          // partial pre of step d+1's entry (row d + 1 - q) over these rows
          const int pn = d + 1 - q;
          float acc = 0.f;
          if (pn >= 0 && pn < TILE) {
            const float4 l0 = *reinterpret_cast<const float4*>(&LBs[pn][i0]);
            const float4 l1 = *reinterpret_cast<const float4*>(&LBs[pn][i0 + 4]);
            acc = fmaf(l0.x, Gg[0], fmaf(l0.y, Gg[1], fmaf(l0.z, Gg[2], l0.w * Gg[3]))) +
                  fmaf(l1.x, Gg[4], fmaf(l1.y, Gg[5], fmaf(l1.z, Gg[6], l1.w * Gg[7])));
            if (g == 0) acc += Xs[pn][q];
          }
          Part[(d + 1) & 1][g][q] = acc;
          __syncthreads();
        }
      }
      // next block: the slot of every column drops by 8, i.e. new slot s = old slot s + 8
      float tmp[TILE];
#pragma unroll
      for (int j = 0; j < TILE; ++j) tmp[j] = LAr[(j + 8) & (TILE - 1)];
#pragma unroll
      for (int j = 0; j < TILE; ++j) LAr[j] = tmp[j];
    }
  }
  // transpose E through a padded buffer (conflict-free both ways)
  for (int e = t; e < TILE * TILE; e += LEAF_THREADS) {
    const int a = e / TILE, b = e % TILE;
    EsT[b][a] = XE[a][b].y;
  }
  __syncthreads();
  for (int e = t; e < TILE * TILE; e += LEAF_THREADS) {
    const int a = e / TILE, b = e % TILE;
    X[(r0 + a) * ldx + c0 + b] = XE[a][b].x;
    if ((r0 + a) < m && (c0 + b) < n) codes[(r0 + a) * n + c0 + b] = Cs[a][b];
    const float ev = EsT[a][b];            // E^T row c0 + a, column r0 + b
    const float hi = tf32_hi(ev);
    const int64_t o = (c0 + a) * ldt + r0 + b;
    EtH[o] = hi;
    EtL[o] = ev - hi;
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
struct TileRegs {
  float v[SIMT_PER];
  __device__ void load(const float* __restrict__ hi, const float* __restrict__ lo, int64_t ld,
                       int64_t row0, int64_t col0, int t) {
#pragma unroll
    for (int k = 0; k < SIMT_PER; ++k) {
      const int e = t + SIMT_THREADS * k;
      const int64_t o = (row0 + e / TILE) * ld + col0 + e % TILE;
      v[k] = hi[o] + lo[o];
    }
  }
  // as stored (S[r][c] = tile[r][c]) or transposed (S[c][r] = tile[r][c])
  __device__ void store(float (*S)[TILE + 1], bool transpose, int t) const {
#pragma unroll
    for (int k = 0; k < SIMT_PER; ++k) {
      const int e = t + SIMT_THREADS * k;
      if (transpose) S[e % TILE][e / TILE] = v[k];
      else S[e / TILE][e % TILE] = v[k];
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

// Stage 1: M[I, J'] = sum_{I' in S1 column J', I' <= I} L^B[I, I'] E[I', J'].
// grid.y walks the rows that have outputs (from row_lo), grid.x the J' span.
__global__ void __launch_bounds__(SIMT_THREADS)
k_band1_simt(Band bd, const float* __restrict__ LBH, const float* __restrict__ LBL, int64_t ldb,
             const float* __restrict__ EtH, const float* __restrict__ EtL, int64_t ldt,
             float* __restrict__ MH, float* __restrict__ ML, int64_t ldm) {
  pdl_wait();
  pdl_trigger();
  const int I = bd.row_lo + blockIdx.y;
  const int jo_hi = bd.jout_hi(I);
  if (bd.jout_lo(I) > jo_hi) return;
  const int Jp = max(0, bd.k - I) + blockIdx.x;
  if (Jp > min(bd.h - 1, jo_hi)) return;
  const int i_lo = max(0, bd.k - Jp), i_hi = min(I, bd.h - 1 - Jp);
  __shared__ float As[TILE][TILE + 1];
  __shared__ float Bs[TILE][TILE + 1];
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  TileRegs ra, rb;
  // B[kk][col] = E[I'*T + kk][J'*T + col] = E^T[J'*T + col][I'*T + kk]
  ra.load(LBH, LBL, ldb, (int64_t)I * TILE, (int64_t)i_lo * TILE, t);
  rb.load(EtH, EtL, ldt, (int64_t)Jp * TILE, (int64_t)i_lo * TILE, t);
  for (int Ip = i_lo; Ip <= i_hi; ++Ip) {
    ra.store(As, false, t);
    rb.store(Bs, true, t);
    __syncthreads();
    if (Ip < i_hi) {
      ra.load(LBH, LBL, ldb, (int64_t)I * TILE, (int64_t)(Ip + 1) * TILE, t);
      rb.load(EtH, EtL, ldt, (int64_t)Jp * TILE, (int64_t)(Ip + 1) * TILE, t);
    }
    tile_mac(As, Bs, tr, tc, acc);
    __syncthreads();
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int64_t o = ((int64_t)I * TILE + tr) * ldm + (int64_t)Jp * TILE + tc + u;
    const float hi = tf32_hi(acc[u]);
    MH[o] = hi;
    ML[o] = acc[u] - hi;
  }
}

// Stage 2: X[I, J] += sum_{J' in [max(0, k - I), min(J, h - 1)]} M[I, J'] L^A[J, J']^T.
__global__ void __launch_bounds__(SIMT_THREADS)
k_band2_simt(Band bd, const float* __restrict__ LAH, const float* __restrict__ LAL, int64_t lda,
             const float* __restrict__ MH, const float* __restrict__ ML, int64_t ldm,
             float* __restrict__ X, int64_t ldx) {
  pdl_wait();
  pdl_trigger();
  const int I = bd.row_lo + blockIdx.y;
  const int J = bd.jout_lo(I) + blockIdx.x;
  if (J > bd.jout_hi(I)) return;
  const int j_lo = max(0, bd.k - I), j_hi = min(J, bd.h - 1);
  __shared__ float As[TILE][TILE + 1];
  __shared__ float Bs[TILE][TILE + 1];   // Bs[t][c] = L^A[J*T + c][J'*T + t]
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  TileRegs ra, rb;
  ra.load(MH, ML, ldm, (int64_t)I * TILE, (int64_t)j_lo * TILE, t);
  rb.load(LAH, LAL, lda, (int64_t)J * TILE, (int64_t)j_lo * TILE, t);
  for (int Jp = j_lo; Jp <= j_hi; ++Jp) {
    ra.store(As, false, t);
    rb.store(Bs, true, t);
    __syncthreads();
    if (Jp < j_hi) {
      ra.load(MH, ML, ldm, (int64_t)I * TILE, (int64_t)(Jp + 1) * TILE, t);
      rb.load(LAH, LAL, lda, (int64_t)J * TILE, (int64_t)(Jp + 1) * TILE, t);
    }
    tile_mac(As, Bs, tr, tc, acc);
    __syncthreads();
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    float* p = X + ((int64_t)I * TILE + tr) * ldx + (int64_t)J * TILE + tc + u;
    *p += acc[u];
  }
}

// Both stages of a narrow node in one launch: each CTA owns one output tile
// (I, J) of S2 and forms the M tiles it needs in shared memory,
//     X[I, J] += sum_{J'} ( sum_{I'} L^B[I, I'] E[I', J'] ) L^A[J, J']^T,
// with the same ranges as the two stages.  Narrow nodes have few (I', J')
// pairs per output, so recomputing an M tile per output costs little and
// saves a launch and the round trip of M through global memory.  The pairs
// are walked as one flat sequence so the next pair's tiles are in flight
// while the current pair is multiplied.
__global__ void __launch_bounds__(SIMT_THREADS)
k_band_fused_simt(Band bd, const float* __restrict__ LBH, const float* __restrict__ LBL,
                  int64_t ldb, const float* __restrict__ EtH, const float* __restrict__ EtL,
                  int64_t ldt, const float* __restrict__ LAH, const float* __restrict__ LAL,
                  int64_t lda, float* __restrict__ X, int64_t ldx) {
  pdl_wait();
  pdl_trigger();
  const int I = bd.row_lo + blockIdx.y;
  const int J = bd.jout_lo(I) + blockIdx.x;
  if (J > bd.jout_hi(I)) return;
  __shared__ float As[TILE][TILE + 1];
  __shared__ float Bs[TILE][TILE + 1];
  __shared__ float Ts[TILE][TILE + 1];
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const int j_lo = max(0, bd.k - I), j_hi = min(J, bd.h - 1);
  auto ilo = [&](int Jp) { return max(0, bd.k - Jp); };
  auto ihi = [&](int Jp) { return min(I, bd.h - 1 - Jp); };
  TileRegs ra, rb, rl;
  int Jp = j_lo, Ip = ilo(j_lo);
  if (Jp <= j_hi) {
    ra.load(LBH, LBL, ldb, (int64_t)I * TILE, (int64_t)Ip * TILE, t);
    rb.load(EtH, EtL, ldt, (int64_t)Jp * TILE, (int64_t)Ip * TILE, t);
    rl.load(LAH, LAL, lda, (int64_t)J * TILE, (int64_t)Jp * TILE, t);
  }
  float m4[4] = {0.f, 0.f, 0.f, 0.f};
  while (Jp <= j_hi) {
    ra.store(As, false, t);
    rb.store(Bs, true, t);
    __syncthreads();
    // next (I', J') pair of the flat walk
    int nJp = Jp, nIp = Ip + 1;
    if (nIp > ihi(Jp)) { nJp = Jp + 1; nIp = nJp <= j_hi ? ilo(nJp) : 0; }
    const bool last_of_col = nJp != Jp;
    if (nJp <= j_hi) {
      ra.load(LBH, LBL, ldb, (int64_t)I * TILE, (int64_t)nIp * TILE, t);
      rb.load(EtH, EtL, ldt, (int64_t)nJp * TILE, (int64_t)nIp * TILE, t);
    }
    tile_mac(As, Bs, tr, tc, m4);
    __syncthreads();
    if (last_of_col) {
      // M[I, J'] complete: multiply by L^A[J, J']^T
#pragma unroll
      for (int u = 0; u < 4; ++u) Ts[tr][tc + u] = m4[u];
      rl.store(Bs, true, t);
      __syncthreads();
      if (nJp <= j_hi) rl.load(LAH, LAL, lda, (int64_t)J * TILE, (int64_t)nJp * TILE, t);
      tile_mac(Ts, Bs, tr, tc, acc);
      __syncthreads();
#pragma unroll
      for (int u = 0; u < 4; ++u) m4[u] = 0.f;
    }
    Jp = nJp;
    Ip = nIp;
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    float* p = X + ((int64_t)I * TILE + tr) * ldx + (int64_t)J * TILE + tc + u;
    *p += acc[u];
  }
}

// ---------------------------------------------------------------- driver
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
  bool tc_ready;
  bool profiling;
  TcOperands tco;
  TcMaps tcm;
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
  if (e != cudaSuccess) a.rc = BAKRON_ERR_CUDA;
}

static void leaf(SolveArgs& a, int K) {
  const int ilo = max(0, K - (a.Nt - 1)), ihi = min(K, a.Mt - 1);
  LaunchScope ls(kFamLeaf, a.s, 2.0 * TILE * TILE * TILE * (ihi - ilo + 1));
  note(a, launch_pdl(k_leaf, dim3(ihi - ilo + 1), dim3(LEAF_THREADS), 0, a.s, K, a.Mt, a.Nt, a.m,
                     a.n, a.X, a.np, a.EtH, a.EtL, a.mp, a.LBH, a.LBL, a.mp, a.LAH, a.LAL, a.np,
                     a.scales, a.zeros, a.G, a.gsz, a.qmax, a.codes, a.status));
}

static void band(SolveArgs& a, int k, int h, int l) {
  double p1 = 0.0, p2 = 0.0;
  if (a.profiling) band_tile_products(a, k, h, l, p1, p2);
  const double f = 2.0 * TILE * TILE * TILE;
  if (a.tc_ready && l - k >= a.tc_min_band) {
    {
      LaunchScope ls(kFamTc1, a.s, f * p1);
      int rc = tc_band_stage(1, a.tcm, a.tco, k, h, l, a.s);
      if (rc != BAKRON_OK) a.rc = rc;
    }
    {
      LaunchScope ls(kFamTc2, a.s, f * p2);
      int rc = tc_band_stage(2, a.tcm, a.tco, k, h, l, a.s);
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
  if (l - k <= a.fused_max_band) {
    LaunchScope ls(kFamFused, a.s, f * (p1 + p2));
    note(a, launch_pdl(k_band_fused_simt, g2, dim3(256), 0, a.s, bd, a.LBH, a.LBL, a.mp, a.EtH,
                       a.EtL, a.mp, a.LAH, a.LAL, a.np, a.X, a.np));
    return;
  }
  {
    LaunchScope ls(kFamBand1, a.s, f * p1);
    note(a, launch_pdl(k_band1_simt, g1, dim3(256), 0, a.s, bd, a.LBH, a.LBL, a.mp, a.EtH,
                       a.EtL, a.mp, a.MH, a.ML, a.np));
  }
  {
    LaunchScope ls(kFamBand2, a.s, f * p2);
    note(a, launch_pdl(k_band2_simt, g2, dim3(256), 0, a.s, bd, a.LAH, a.LAL, a.np, a.MH, a.ML,
                       a.np, a.X, a.np));
  }
}

static void rec(SolveArgs& a, int k, int l) {
  if (l == k + 1) {
    leaf(a, k);
    return;
  }
  const int h = (k + l) / 2;
  rec(a, k, h);
  band(a, k, h, l);
  rec(a, h, l);
}

int solve_impl(const void* W, int wdt, int m, int n, int64_t ldw, const void* factors, int bits,
               int group_size, uint8_t* codes, float* scales, float* zeros, float* prerounding,
               void* workspace, cudaStream_t s) {
  FactorLayout fl(m, n);
  SolveLayout sl(m, n);
  char* ws = (char*)workspace;
  const char* f = (const char*)factors;
  SolveArgs a;
  a.m = m; a.n = n;
  a.Mt = ceil_div(m, TILE); a.Nt = ceil_div(n, TILE);
  a.gsz = group_size == 0 ? n : group_size;
  a.G = n / a.gsz;
  a.qmax = (1 << bits) - 1;
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
  a.profiling = profiling_on();
  {
    const char* e = getenv("BAKRON_TC_MIN_BAND");
    a.tc_min_band = (e && *e) ? atoi(e) : 16;   // 0 or less: tensor cores off
    const char* f2 = getenv("BAKRON_FUSED_MAX_BAND");
    a.fused_max_band = (f2 && *f2) ? atoi(f2) : 4;
    a.tc_ready = false;
    if (a.tc_min_band > 0) {
      a.tco = TcOperands{a.mp, a.np, a.Mt, a.Nt, a.LBH, a.LBL, a.LAH, a.LAL,
                         a.EtH, a.EtL, a.MH, a.ML, a.X, a.status};
      a.tc_ready = tc_band_maps(a.tcm, a.tco);
      if (!a.tc_ready) return BAKRON_ERR_CUDA;
    }
  }
  reset_launch_count();
  BK_CUDA_OK(cudaMemsetAsync(ws + sl.off_status, 0, 256, s));
  {
    const int64_t warps = (int64_t)m * a.G;
    LaunchScope ls(kFamInit, s);
    k_grid<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, s>>>(W, wdt, m, n, ldw, a.gsz, a.G,
                                                                 a.qmax, scales, zeros);
  }
  {
    const int64_t tot = a.mp * a.np;
    LaunchScope ls(kFamInit, s);
    note(a, launch_pdl(k_init, dim3((unsigned)((tot + 255) / 256)), dim3(256), 0, s, W, wdt, m, n,
                       ldw, a.X, a.mp, a.np));
  }
  rec(a, 0, a.Mt + a.Nt - 1);
  if (prerounding) {
    const int64_t tot = (int64_t)m * n;
    LaunchScope ls(kFamCopy, s);
    note(a, launch_pdl(k_copy_out, dim3((unsigned)((tot + 255) / 256)), dim3(256), 0, s,
                       (const float*)a.X, a.np, m, n, prerounding));
  }
  BK_CUDA_OK(cudaGetLastError());
  return a.rc;
}

}  // namespace bakron
