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
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= (int64_t)m * n) return;
  const int64_t r = idx / n, c = idx % n;
  out[idx] = X[r * np + c];
}

// ------------------------------------------------------------------ leaf
// One CTA rounds one TILE x TILE tile whose inbound updates from all earlier
// tiles are already in X (paper, the parallel anti-diagonal loop of Sec. 3.3,
// run inside the tile).  Four warps stage the tile, its factor blocks and its
// grid in shared memory; warp 0 then walks the 63 anti-diagonals.  Lane q owns
// column q; at in-tile step d it rounds entry (p, q), p = d - q.  Intra-tile
// feedback is factored as
//     x_pq = X_pq + sum_i L^B[p][i] G_q[i],   G_q[i] = sum_{j<=q} e_ij L^A[q][j]
// where G_q[i] only ever holds errors already committed: for i < p all of row
// i up to column q (committed at steps i + j < d), for i = p the columns
// j < q, and rows i > p are multiplied by L^B[p][i] = 0.  L^B[p][p] = 1 adds
// G_q[p] itself.  Each step's errors are broadcast through shared memory and
// folded into G with register indices fixed at compile time (d, j unrolled).
// Outputs: codes, X (pre-rounding values) and E^T as a tf32 hi/lo pair.
constexpr int LEAF_THREADS = 128;

__global__ void __launch_bounds__(LEAF_THREADS)
k_leaf(int K, int Mt, int Nt, int m, int n, float* __restrict__ X, int64_t ldx,
       float* __restrict__ EtH, float* __restrict__ EtL, int64_t ldt,
       const float* __restrict__ LBH, const float* __restrict__ LBL, int64_t ldb,
       const float* __restrict__ LAH, const float* __restrict__ LAL, int64_t lda,
       const float* __restrict__ scales, const float* __restrict__ zeros, int G, int gsz,
       int qmax, uint8_t* __restrict__ codes, int* status) {
  const int I = max(0, K - (Nt - 1)) + blockIdx.x;
  const int J = K - I;
  const int t = threadIdx.x;
  __shared__ float Xs[TILE][TILE];              // stride 32: anti-diagonal access hits 32 banks
  __shared__ __align__(16) float LBs[TILE][36];  // stride 36: conflict-free float4 row reads
  __shared__ float LAs[TILE][TILE + 1];
  __shared__ float St[TILE][TILE], Zt[TILE][TILE];
  __shared__ float Es[TILE][TILE];
  __shared__ __align__(16) float Eb[2][TILE];
  const int64_t r0 = (int64_t)I * TILE, c0 = (int64_t)J * TILE;
#pragma unroll
  for (int k = 0; k < TILE * TILE / LEAF_THREADS; ++k) {
    const int e = t + k * LEAF_THREADS;
    const int p = e / TILE, c = e % TILE;
    Xs[p][c] = X[(r0 + p) * ldx + c0 + c];
    const int64_t ob = (r0 + p) * ldb + r0 + c, oa = (c0 + p) * lda + c0 + c;
    LBs[p][c] = LBH[ob] + LBL[ob];
    LAs[p][c] = LAH[oa] + LAL[oa];
    const bool real = (r0 + p) < m && (c0 + c) < n;
    const int64_t og = (r0 + p) * G + (c0 + c) / gsz;
    St[p][c] = real ? scales[og] : 1.f;
    Zt[p][c] = real ? zeros[og] : 0.f;
  }
  __syncthreads();
  if (t < 32) {
    const int q = t;
    const bool col_real = (c0 + q) < n;
    float LAr[TILE];
#pragma unroll
    for (int j = 0; j < TILE; ++j) LAr[j] = LAs[q][j];
    float Gq[TILE];
#pragma unroll
    for (int i = 0; i < TILE; ++i) Gq[i] = 0.f;
    const float fq = (float)qmax;
    bool bad = false;
#pragma unroll
    for (int d = 0; d < 2 * TILE - 1; ++d) {
      const int p = d - q;
      const bool act = p >= 0 && p < TILE;
      const int pc = act ? p : 0;
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
      for (int i = 0; i < TILE; i += 4) {
        if (i > d) break;  // rows below d hold no committed error yet
        const float4 l = *reinterpret_cast<const float4*>(&LBs[pc][i]);
        a0 = fmaf(l.x, Gq[i], a0);
        a1 = fmaf(l.y, Gq[i + 1], a1);
        a2 = fmaf(l.z, Gq[i + 2], a2);
        a3 = fmaf(l.w, Gq[i + 3], a3);
      }
      float e = 0.f;
      if (act) {
        const float x = Xs[pc][q] + ((a0 + a1) + (a2 + a3));
        const float s = St[pc][q], z = Zt[pc][q];
        float c = rintf(__fdiv_rn(x, s)) + z;
        c = fminf(fmaxf(c, 0.f), fq);
        const float v = __fmul_rn(s, __fsub_rn(c, z));
        e = __fsub_rn(v, x);
        const bool real = (r0 + p) < m && col_real;
        if (!real) e = 0.f;
        else codes[(r0 + p) * n + c0 + q] = (uint8_t)c;
        bad |= !isfinite(x);
        Xs[pc][q] = x;
        Es[pc][q] = e;
      }
      Eb[d & 1][q] = e;
      __syncwarp();
#pragma unroll
      for (int j4 = 0; j4 < TILE; j4 += 4) {
        if (d - j4 - 3 >= TILE || d - j4 < 0) continue;  // no row of this group on step d
        const float4 ev = *reinterpret_cast<const float4*>(&Eb[d & 1][j4]);
        const float evs[4] = {ev.x, ev.y, ev.z, ev.w};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = d - (j4 + u);
          if (i >= 0 && i < TILE) Gq[i] = fmaf(evs[u], LAr[j4 + u], Gq[i]);
        }
      }
    }
    if (bad) raise_status(status, BAKRON_ERR_NONFINITE);
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < TILE * TILE / LEAF_THREADS; ++k) {
    const int e = t + k * LEAF_THREADS;
    const int a = e / TILE, b = e % TILE;
    X[(r0 + a) * ldx + c0 + b] = Xs[a][b];
    const float ev = Es[b][a];             // E^T row c0 + a, column r0 + b
    const float hi = tf32_hi(ev);
    const int64_t o = (c0 + a) * ldt + r0 + b;
    EtH[o] = hi;
    EtL[o] = ev - hi;
  }
}

// ------------------------------------------------------- band products (SIMT)
// 32 x 32 output tile per CTA, 256 threads, 4 outputs each.  Both stages
// derive their tile ranges from (k, h, l) in closed form.
struct Band {
  int k, h, l, Mt, Nt;
  __host__ __device__ int jout_lo(int I) const { return max(0, h - I); }
  __host__ __device__ int jout_hi(int I) const { return min(Nt - 1, l - 1 - I); }
};

// Stage 1: M[I, J'] = sum_{I' in S1 column J', I' <= I} L^B[I, I'] E[I', J'].
__global__ void __launch_bounds__(256)
k_band1_simt(Band bd, const float* __restrict__ LBH, const float* __restrict__ LBL, int64_t ldb,
             const float* __restrict__ EtH, const float* __restrict__ EtL, int64_t ldt,
             float* __restrict__ MH, float* __restrict__ ML, int64_t ldm) {
  const int I = blockIdx.y;
  const int jo_hi = bd.jout_hi(I);
  if (bd.jout_lo(I) > jo_hi) return;
  const int Jp = max(0, bd.k - I) + blockIdx.x;
  if (Jp > min(bd.h - 1, jo_hi)) return;
  const int i_lo = max(0, bd.k - Jp), i_hi = min(I, bd.h - 1 - Jp);
  __shared__ float As[TILE][TILE + 1];
  __shared__ float Bs[TILE][TILE + 1];
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int Ip = i_lo; Ip <= i_hi; ++Ip) {
    for (int e = t; e < TILE * TILE; e += 256) {
      const int r = e / TILE, c = e % TILE;
      const int64_t oa = ((int64_t)I * TILE + r) * ldb + (int64_t)Ip * TILE + c;
      As[r][c] = LBH[oa] + LBL[oa];
      // B[kk][col] = E[Ip*T + kk][Jp*T + col] = E^T[Jp*T + col][Ip*T + kk]
      const int64_t ob = ((int64_t)Jp * TILE + r) * ldt + (int64_t)Ip * TILE + c;
      Bs[c][r] = EtH[ob] + EtL[ob];
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < TILE; ++kk) {
      const float a = As[tr][kk];
#pragma unroll
      for (int u = 0; u < 4; ++u) acc[u] = fmaf(a, Bs[kk][tc + u], acc[u]);
    }
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
__global__ void __launch_bounds__(256)
k_band2_simt(Band bd, const float* __restrict__ LAH, const float* __restrict__ LAL, int64_t lda,
             const float* __restrict__ MH, const float* __restrict__ ML, int64_t ldm,
             float* __restrict__ X, int64_t ldx) {
  const int I = blockIdx.y;
  const int J = bd.jout_lo(I) + blockIdx.x;
  if (J > bd.jout_hi(I)) return;
  const int j_lo = max(0, bd.k - I), j_hi = min(J, bd.h - 1);
  __shared__ float As[TILE][TILE + 1];
  __shared__ float Bs[TILE][TILE + 1];   // Bs[t][c] = L^A[J*T + c][J'*T + t]
  const int t = threadIdx.x, tr = t / 8, tc = (t % 8) * 4;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int Jp = j_lo; Jp <= j_hi; ++Jp) {
    for (int e = t; e < TILE * TILE; e += 256) {
      const int r = e / TILE, c = e % TILE;
      const int64_t om = ((int64_t)I * TILE + r) * ldm + (int64_t)Jp * TILE + c;
      As[r][c] = MH[om] + ML[om];
      const int64_t oa = ((int64_t)J * TILE + r) * lda + (int64_t)Jp * TILE + c;
      Bs[c][r] = LAH[oa] + LAL[oa];
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < TILE; ++kk) {
      const float a = As[tr][kk];
#pragma unroll
      for (int u = 0; u < 4; ++u) acc[u] = fmaf(a, Bs[kk][tc + u], acc[u]);
    }
    __syncthreads();
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
  bool tc_ready;
  TcOperands tco;
  TcMaps tcm;
  int rc;
};

static void leaf(const SolveArgs& a, int K) {
  const int ilo = max(0, K - (a.Nt - 1)), ihi = min(K, a.Mt - 1);
  LaunchScope ls(kFamLeaf, a.s);
  k_leaf<<<ihi - ilo + 1, LEAF_THREADS, 0, a.s>>>(
      K, a.Mt, a.Nt, a.m, a.n, a.X, a.np, a.EtH, a.EtL, a.mp, a.LBH, a.LBL, a.mp, a.LAH, a.LAL,
      a.np, a.scales, a.zeros, a.G, a.gsz, a.qmax, a.codes, a.status);
}

static void band(SolveArgs& a, int k, int h, int l) {
  if (a.tc_ready && l - k >= a.tc_min_band) {
    {
      LaunchScope ls(kFamBand1, a.s);
      int rc = tc_band_stage(1, a.tcm, a.tco, k, h, l, a.s);
      if (rc != BAKRON_OK) a.rc = rc;
    }
    {
      LaunchScope ls(kFamBand2, a.s);
      int rc = tc_band_stage(2, a.tcm, a.tco, k, h, l, a.s);
      if (rc != BAKRON_OK) a.rc = rc;
    }
    return;
  }
  Band bd{k, h, l, a.Mt, a.Nt};
  dim3 g1(h, a.Mt), g2(l - h, a.Mt);
  {
    LaunchScope ls(kFamBand1, a.s);
    k_band1_simt<<<g1, 256, 0, a.s>>>(bd, a.LBH, a.LBL, a.mp, a.EtH, a.EtL, a.mp, a.MH, a.ML,
                                      a.np);
  }
  {
    LaunchScope ls(kFamBand2, a.s);
    k_band2_simt<<<g2, 256, 0, a.s>>>(bd, a.LAH, a.LAL, a.np, a.MH, a.ML, a.np, a.X, a.np);
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
  {
    const char* e = getenv("BAKRON_TC_MIN_BAND");
    a.tc_min_band = (e && *e) ? atoi(e) : 16;   // 0 or less: tensor cores off
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
    k_init<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(W, wdt, m, n, ldw, a.X, a.mp, a.np);
  }
  rec(a, 0, a.Mt + a.Nt - 1);
  if (a.rc != BAKRON_OK) return a.rc;
  if (prerounding) {
    const int64_t tot = (int64_t)m * n;
    LaunchScope ls(kFamCopy, s);
    k_copy_out<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(a.X, a.np, m, n, prerounding);
  }
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}

}  // namespace bakron
