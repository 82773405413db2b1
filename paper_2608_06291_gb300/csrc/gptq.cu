// The B = I case of the solve (GPTQ, Sec. 1 and Alg. 1): with L^B = I the
// rows of W are independent, entry (p, q) depends only on the entries left of
// it in its own row, and the two-sided recursion collapses to column splits
// (Alg. 4 splitting columns only):
//
//   rec(c0, c1): a range of at most GQ_BLOCK tile columns is a leaf launch;
//                otherwise h = (c0 + c1) / 2, rec(c0, h),
//                X[:, h..c1) += E[:, c0..h) L^A[h..c1, c0..h)^T  (tensor cores),
//                rec(h, c1).
//
// A leaf launch gives one CTA to each 32-row strip of W; its first warp (lane
// p = row p) walks the range's columns in order, the other three write the
// finished tiles out and help form the windows.  Column q of a tile is one
// step: every lane rounds its row's entry, x_pq -> code, e_pq = s (c - z) - x,
// then adds e_pq L^A[q'][q] to the pre-rounding values of the later columns
// q' of the tile, which it keeps in registers.  A later tile of the range
// starts from X plus the errors of the range's earlier tiles times the
// matching blocks of L^A (the Alg. 4 nodes inside the range).  So a tile of
// 32 x 32 entries takes 32 dependent steps, and all strips run side by side.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdlib>
#include <mutex>

#include "common.cuh"
#include "profile.cuh"
#include "tc_gemm.cuh"
#include "tune.cuh"

namespace bakron {

constexpr int GQ_BLOCK = 4;                               // tile columns per leaf launch
constexpr int GQ_THREADS = 128;                           // warp 0 rounds; all four form windows
constexpr int GQ_LA_BLOCKS = GQ_BLOCK * (GQ_BLOCK + 1) / 2;   // L^A blocks one launch reads

struct GptqArgs {
  int Mt, Nt, m, n;
  float* X;                     // pre-rounding values, in place (mp x np, row stride ldx)
  int64_t ldx;
  float *EH, *EL;               // E as tf32 hi / lo, row-major like X (the column band's A)
  const float* LAblk;           // the factor buffer's L^A leaf blocks
  const float *scales, *zeros;
  int G, gsz, qmax;
  uint8_t* codes;
  int* status;
  unsigned long long* stamp;
};

struct GptqSmem {
  // L^A[J, J - g] of every tile J of the range and g = 0 .. J - c0, k-major
  // ([j][q] = L^A[J, J-g][q][j]), in the order (J - c0) (J - c0 + 1) / 2 + g
  __align__(16) float LA[GQ_LA_BLOCKS][TILE][LEAF_BLOCK_LD];
  // X of the strip's range, copied in with 16-byte asynchronous copies (rows
  // 132 floats apart: 16-byte aligned, and the float4 reads of 8 lanes of
  // different rows fall in different banks)
  __align__(16) float Xin[TILE][GQ_BLOCK * TILE + 4];
  float Xo[TILE][GQ_BLOCK * TILE + 1];   // pre-rounding values out
  float Es[GQ_BLOCK][TILE][TILE + 1];    // errors of the range's tiles, [p][j]
  float T1[TILE][TILE + 1];              // the window's sum for the current tile, [p][q]
  uint8_t Cs[TILE][GQ_BLOCK * TILE + 4]; // codes (rows 132 bytes apart: no bank conflicts)
};

__device__ __forceinline__ void gq_cp_async16(void* dst, const void* src) {
  const unsigned d = (unsigned)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
}

// Part of the window of tile t of the range: the sum over g = g0 .. g1 of
// E[I, J-g] L^A[J, J-g]^T (fp32-accurate by the 3xTF32 split), columns
// 8 ni0 .. 8 (ni0 + NI) - 1, stored into dst ([p][q]) plus `base` when given.
// With lane = 4 gid + tig, an m16n8k8 fragment holds A(gid (+8), tig (+4)),
// B(k = tig (+4), n = gid) and D(gid (+8), 2 tig (+1)).
template <int NI>
__device__ __forceinline__ void gptq_window(const GptqSmem& S, int t, int g0, int g1, int ni0,
                                            const float (*base)[TILE + 1], float (*dst)[TILE + 1],
                                            int lane) {
  const int gid = lane >> 2, tig = lane & 3;
  float d[2][NI][4];
#pragma unroll
  for (int mi = 0; mi < 2; ++mi)
#pragma unroll
    for (int ni = 0; ni < NI; ++ni)
#pragma unroll
      for (int r = 0; r < 4; ++r) d[mi][ni][r] = 0.f;
  for (int g = g0; g <= g1; ++g) {
    const float(*Lg)[LEAF_BLOCK_LD] = S.LA[t * (t + 1) / 2 + g];   // B(k = j, n = q) = Lg[j][q]
    const float(*Eg)[TILE + 1] = S.Es[t - g];                       // A(p, j) = Eg[p][j]
#pragma unroll
    for (int kk = 0; kk < TILE / 8; ++kk) {
      uint32_t ah[2][4], al[2][4], bh[NI][2], bl[NI][2];
#pragma unroll
      for (int mi = 0; mi < 2; ++mi) {
        const int r = 16 * mi + gid, c = 8 * kk + tig;
        tf32_split(Eg[r][c], ah[mi][0], al[mi][0]);
        tf32_split(Eg[r + 8][c], ah[mi][1], al[mi][1]);
        tf32_split(Eg[r][c + 4], ah[mi][2], al[mi][2]);
        tf32_split(Eg[r + 8][c + 4], ah[mi][3], al[mi][3]);
      }
#pragma unroll
      for (int ni = 0; ni < NI; ++ni) {
        const int k = 8 * kk + tig, n = 8 * (ni0 + ni) + gid;
        tf32_split(Lg[k][n], bh[ni][0], bl[ni][0]);
        tf32_split(Lg[k + 4][n], bh[ni][1], bl[ni][1]);
      }
#pragma unroll
      for (int mi = 0; mi < 2; ++mi)
#pragma unroll
        for (int ni = 0; ni < NI; ++ni) {
          mma_tf32_16x8x8(d[mi][ni], al[mi], bh[ni]);
          mma_tf32_16x8x8(d[mi][ni], ah[mi], bl[ni]);
          mma_tf32_16x8x8(d[mi][ni], ah[mi], bh[ni]);
        }
    }
  }
#pragma unroll
  for (int mi = 0; mi < 2; ++mi)
#pragma unroll
    for (int ni = 0; ni < NI; ++ni) {
      const int r = 16 * mi + gid, c = 8 * (ni0 + ni) + 2 * tig;
      dst[r][c] = d[mi][ni][0] + (base ? base[r][c] : 0.f);
      dst[r][c + 1] = d[mi][ni][1] + (base ? base[r][c + 1] : 0.f);
      dst[r + 8][c] = d[mi][ni][2] + (base ? base[r + 8][c] : 0.f);
      dst[r + 8][c + 1] = d[mi][ni][3] + (base ? base[r + 8][c + 1] : 0.f);
    }
}

// The outputs of tile t of the range from shared memory, by `nthr` threads
// numbered from tid: pre-rounding values, codes, and E as an exact tf32
// hi/lo pair for the column band (row by row, 32 consecutive columns per warp).
__device__ __forceinline__ void gptq_store_tile(const GptqSmem& S, const GptqArgs& a, int64_t r0,
                                                int64_t cbase, int t, int tid, int nthr) {
  for (int e = tid; e < TILE * TILE; e += nthr) {
    const int i = e / TILE, c = e % TILE;
    const int64_t r = r0 + i, col = cbase + (int64_t)t * TILE + c;
    const int64_t o = r * a.ldx + col;
    a.X[o] = S.Xo[i][t * TILE + c];
    const float ev = S.Es[t][i][c];
    const float hi = tf32_hi(ev);
    a.EH[o] = hi;
    a.EL[o] = ev - hi;
    if (r < a.m && col < a.n) a.codes[r * a.n + col] = S.Cs[i][t * TILE + c];
  }
}

// Tiles c0 .. c0 + nt - 1 (nt <= GQ_BLOCK) of the strip of tile row blockIdx.x.
// Warp 0 walks the columns (lane = row); per tile, all four warps first form
// its window (one 8-column slice each), then, while warp 0 rounds the tile,
// warps 1-3 write the previous tile's outputs.  Every thread passes the same
// CTA barriers.
__global__ void __launch_bounds__(GQ_THREADS) k_gptq_leaf(int c0, int nt, GptqArgs a) {
  extern __shared__ __align__(16) unsigned char gq_smem[];
  GptqSmem& S = *reinterpret_cast<GptqSmem*>(gq_smem);
  const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31;
  const int p = lane;                   // warp 0: row of the strip
  const int I = blockIdx.x;
  const int64_t r0 = (int64_t)I * TILE, cbase = (int64_t)c0 * TILE;
  // factor blocks (read-only during the solve) before waiting for the
  // previous kernel
  for (int t = 0; t < nt; ++t)
    for (int g = 0; g <= t; ++g) {
      const float* src = a.LAblk + ((int64_t)(c0 + t) * LEAF_BLOCKS + g) * LEAF_BLOCK_FLOATS;
      float* dst = &S.LA[t * (t + 1) / 2 + g][0][0];
      for (int c = tid; c < LEAF_BLOCK_FLOATS / 4; c += GQ_THREADS)
        gq_cp_async16(dst + 4 * c, src + 4 * c);
    }
  asm volatile("cp.async.commit_group;" ::: "memory");
  // this row's grid on each tile (a group covers whole tiles: gsz % 32 == 0)
  const int64_t row = r0 + p;
  const bool row_real = row < a.m;
  float sv[GQ_BLOCK], iv[GQ_BLOCK], zv[GQ_BLOCK];
#pragma unroll
  for (int t = 0; t < GQ_BLOCK; ++t) {
    const int64_t col = cbase + (int64_t)t * TILE;
    const bool ok = w == 0 && row_real && t < nt && col < a.n;
    const float s = ok ? a.scales[row * a.G + col / a.gsz] : 1.f;
    sv[t] = s;
    iv[t] = 1.f / s;
    zv[t] = ok ? a.zeros[row * a.G + col / a.gsz] : 0.f;
  }
  pdl_wait();
  pdl_trigger();
  stamp_begin(a.stamp);
  // X of the strip's range: all its 16-byte chunks in flight at once
  const int chunks_per_row = nt * TILE / 4;
  for (int c = tid; c < TILE * chunks_per_row; c += GQ_THREADS) {
    const int i = c / chunks_per_row, k = c % chunks_per_row;
    gq_cp_async16(&S.Xin[i][4 * k], a.X + (r0 + i) * a.ldx + cbase + 4 * k);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();

  constexpr float R = 12582912.f;   // 1.5 * 2^23: fl(v + R) - R rounds v to an integer
  const float fq = (float)a.qmax;
  bool bad = false;
  for (int t = 0; t < nt; ++t) {
    // T1 = the window of tile t, one 8-column slice per warp, every entry
    // summed over g = 1 .. t in that order
    if (t >= 1) gptq_window<1>(S, t, 1, t, w, nullptr, S.T1, lane);
    __syncthreads();   // S.T1 complete
    if (w == 0) {
      const int64_t col0 = cbase + (int64_t)t * TILE;
      float acc[TILE];
#pragma unroll
      for (int q4 = 0; q4 < TILE / 4; ++q4) {
        const float4 v = *reinterpret_cast<const float4*>(&S.Xin[p][t * TILE + 4 * q4]);
        acc[4 * q4] = v.x;
        acc[4 * q4 + 1] = v.y;
        acc[4 * q4 + 2] = v.z;
        acc[4 * q4 + 3] = v.w;
      }
      if (t >= 1) {
#pragma unroll
        for (int q = 0; q < TILE; ++q) acc[q] += S.T1[p][q];
      }
      // the tile's 32 steps; the unit diagonal of L^A[J, J] is this entry's own.
      // Row q + 1 of L^A[J, J] is read into registers during step q, before
      // that step's shared-memory stores, so its loads are never waited for.
      const float(*L0)[LEAF_BLOCK_LD] = S.LA[t * (t + 1) / 2];
      const float s = sv[t], inv = iv[t], mz = -zv[t];
      float4 Lc[TILE / 4], Ln[TILE / 4];
#pragma unroll
      for (int q4 = 0; q4 < TILE / 4; ++q4) {
        Lc[q4] = *reinterpret_cast<const float4*>(&L0[0][4 * q4]);
        Ln[q4] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int q = 0; q < TILE; ++q) {
        if (q + 1 < TILE) {
#pragma unroll
          for (int q4 = (q + 2) / 4; q4 < TILE / 4; ++q4)
            Ln[q4] = *reinterpret_cast<const float4*>(&L0[q + 1][4 * q4]);
        }
        const float x = acc[q];
        const float tc = fminf(fmaxf(fmaf(x, inv, R), R + mz), R + fq + mz);
        const float mk = (row_real && col0 + q < a.n) ? 1.f : 0.f;
        const float e = fmaf(s * mk, tc - R, x * -mk);   // s (c - z) - x, rounded once
#pragma unroll
        for (int q4 = (q + 1) / 4; q4 < TILE / 4; ++q4) {
          const float4 l = Lc[q4];
          if (4 * q4 > q) acc[4 * q4] = fmaf(e, l.x, acc[4 * q4]);
          if (4 * q4 + 1 > q) acc[4 * q4 + 1] = fmaf(e, l.y, acc[4 * q4 + 1]);
          if (4 * q4 + 2 > q) acc[4 * q4 + 2] = fmaf(e, l.z, acc[4 * q4 + 2]);
          if (4 * q4 + 3 > q) acc[4 * q4 + 3] = fmaf(e, l.w, acc[4 * q4 + 3]);
        }
        bad |= !isfinite(x);
        S.Xo[p][t * TILE + q] = x;
        S.Es[t][p][q] = e;
        S.Cs[p][t * TILE + q] = (uint8_t)(int)(tc - (R + mz));
#pragma unroll
        for (int q4 = 0; q4 < TILE / 4; ++q4) Lc[q4] = Ln[q4];
      }
    } else if (t >= 1) {
      gptq_store_tile(S, a, r0, cbase, t - 1, tid - 32, GQ_THREADS - 32);
    }
    __syncthreads();   // tile t's values, errors and codes in shared memory
  }
  gptq_store_tile(S, a, r0, cbase, nt - 1, tid, GQ_THREADS);
  if (bad) raise_status(a.status, BAKRON_ERR_NONFINITE);
  stamp_end(a.stamp);
}

namespace {
struct GqRun {
  GptqArgs la;
  TcMaps tcm;
  TcOperands tco;
  cudaStream_t s;
  int rc;
};

void gq_leaf(GqRun& r, int c0, int c1) {
  LaunchScope ls(kFamLeaf, r.s, 2.0 * TILE * TILE * TILE * r.la.Mt * (c1 - c0) * (c1 - c0 + 1) / 2);
  GptqArgs la = r.la;
  la.stamp = ls.stamp();
  const cudaError_t e = launch_pdl(k_gptq_leaf, dim3(r.la.Mt), dim3(GQ_THREADS), sizeof(GptqSmem),
                                   r.s, c0, c1 - c0, la);
  if (e != cudaSuccess) r.rc = cuda_fail(e, __FILE__, __LINE__);
}

void gq_rec(GqRun& r, int c0, int c1) {
  if (c1 - c0 <= GQ_BLOCK) {
    gq_leaf(r, c0, c1);
    return;
  }
  const int h = (c0 + c1) / 2;
  gq_rec(r, c0, h);
  {
    LaunchScope ls(kFamTc2, r.s, 2.0 * TILE * TILE * TILE * r.la.Mt * (h - c0) * (c1 - h));
    const int rc = tc_cols_stage(r.tcm, r.tco, c0, h, c1, r.s, ls.stamp());
    if (rc != BAKRON_OK) r.rc = rc;
  }
  gq_rec(r, h, c1);
}
}  // namespace

int launch_solve_prologue(const void* W, int wdt, int m, int n, int64_t ldw, int gsz, int G,
                          int qmax, float* scales, float* zeros, float* X, int64_t mp, int64_t np,
                          char* status_area, cudaStream_t s);
int launch_copy_out(const float* X, int64_t np, int m, int n, float* out, cudaStream_t s);

int gptq_impl(const void* W, int wdt, int m, int n, int64_t ldw, const void* factors, int qmax,
              int group_size, uint8_t* codes, float* scales, float* zeros, float* prerounding,
              void* workspace, cudaStream_t s) {
  FactorLayout fl(m, n);
  SolveLayout sl(m, n);
  char* ws = (char*)workspace;
  const char* f = (const char*)factors;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(k_gptq_leaf, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)sizeof(GptqSmem));
  });
  if (attr_err != cudaSuccess) return BAKRON_ERR_CUDA;
  GqRun r;
  r.s = s;
  r.rc = BAKRON_OK;
  const int Mt = ceil_div(m, TILE), Nt = ceil_div(n, TILE);
  const int gsz = group_size == 0 ? n : group_size;
  float* X = (float*)(ws + sl.off_X);
  float* MH = (float*)(ws + sl.off_MH);
  float* ML = (float*)(ws + sl.off_ML);
  int* status = (int*)(ws + sl.off_status);
  r.la = GptqArgs{Mt, Nt, m, n, X, sl.np, MH, ML, (const float*)(f + fl.off_LAblk), scales,
                  zeros, n / gsz, gsz, qmax, codes, status, nullptr};
  r.tco = TcOperands{sl.mp, sl.np, Mt, Nt,
                     (const float*)(f + fl.off_LBH), (const float*)(f + fl.off_LBL),
                     (const float*)(f + fl.off_LAH), (const float*)(f + fl.off_LAL),
                     (float*)(ws + sl.off_EtH), (float*)(ws + sl.off_EtL), MH, ML, X, status};
  if (!tc_band_maps(r.tcm, r.tco)) return BAKRON_ERR_CUDA;
  reset_launch_count();
  int rc = launch_solve_prologue(W, wdt, m, n, ldw, gsz, n / gsz, qmax, scales, zeros, X, sl.mp,
                                 sl.np, ws + sl.off_status, s);
  if (rc != BAKRON_OK) return rc;
  gq_rec(r, 0, Nt);
  if (prerounding) {
    rc = launch_copy_out(X, sl.np, m, n, prerounding, s);
    if (rc != BAKRON_OK) return rc;
  }
  BK_CUDA_OK(cudaGetLastError());
  return r.rc;
}

}  // namespace bakron
