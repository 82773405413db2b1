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
// One warp rounds one TILE x TILE tile whose inbound updates from all earlier
// tiles are already in X (paper, Alg. 3's parallel anti-diagonal step, run
// inside the tile).  Lane q owns column q; at in-tile step d it rounds entry
// (p, q), p = d - q.  Intra-tile feedback is factored as
//     x_pq = X_pq + sum_i L^B[p][i] G_q[i],   G_q[i] = sum_{j<=q} e_ij L^A[q][j]
// where G_q[i] only ever holds errors already committed: for i < p all of row
// i up to column q (committed at steps i + j < d), for i = p the columns
// j < q, and rows i > p are multiplied by L^B[p][i] = 0.  L^B[p][p] = 1 adds
// G_q[p] itself.  Each step's errors are broadcast through shared memory and
// folded into G with register indices fixed at compile time (d, j unrolled).
__global__ void __launch_bounds__(32)
k_leaf(int K, int Mt, int Nt, int m, int n, float* __restrict__ X, float* __restrict__ E,
       int64_t ldx, const float* __restrict__ LB, int64_t ldb, const float* __restrict__ LA,
       int64_t lda, const float* __restrict__ scales, const float* __restrict__ zeros, int G,
       int gsz, int qmax, uint8_t* __restrict__ codes, int* status) {
  const int I = max(0, K - (Nt - 1)) + blockIdx.x;
  const int J = K - I;
  const int q = threadIdx.x;
  __shared__ float Xs[TILE][TILE];              // stride 32: anti-diagonal reads hit 32 banks
  __shared__ __align__(16) float LBs[TILE][36];  // stride 36: conflict-free float4 row reads
  __shared__ float St[TILE][TILE], Zt[TILE][TILE];
  __shared__ float Es[TILE][TILE];
  __shared__ __align__(16) float Eb[2][TILE];
  const int64_t r0 = (int64_t)I * TILE, c0 = (int64_t)J * TILE;
  const int gq = (int)((c0 + q) / gsz);
  const bool col_real = (c0 + q) < n;
#pragma unroll 4
  for (int p = 0; p < TILE; ++p) {
    Xs[p][q] = X[(r0 + p) * ldx + c0 + q];
    LBs[p][q] = LB[(r0 + p) * ldb + r0 + q];
    const bool real = (r0 + p) < m && col_real;
    St[p][q] = real ? scales[(r0 + p) * G + gq] : 1.f;
    Zt[p][q] = real ? zeros[(r0 + p) * G + gq] : 0.f;
  }
  float LAr[TILE];
  {
    const float4* src = reinterpret_cast<const float4*>(LA + (c0 + q) * lda + c0);
#pragma unroll
    for (int j = 0; j < TILE / 4; ++j) {
      float4 v = src[j];
      LAr[4 * j] = v.x; LAr[4 * j + 1] = v.y; LAr[4 * j + 2] = v.z; LAr[4 * j + 3] = v.w;
    }
  }
  float Gq[TILE];
#pragma unroll
  for (int i = 0; i < TILE; ++i) Gq[i] = 0.f;
  __syncwarp();
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
      // rows above d can hold no committed error yet: skip at compile time
      if (i > d) break;
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
      if (d - j4 - 3 >= TILE || d - j4 < 0) continue;   // no row of this group on step d
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
  __syncwarp();
#pragma unroll 4
  for (int p = 0; p < TILE; ++p) {
    X[(r0 + p) * ldx + c0 + q] = Xs[p][q];
    E[(r0 + p) * ldx + c0 + q] = Es[p][q];
  }
}

// ------------------------------------------------------- band products (SIMT)
// 32 x 32 output tile per CTA, 256 threads, 4 outputs each.  Both stages
// derive their tile ranges from (k, h, l) in closed form.
struct Band {
  int k, h, l, Mt, Nt;
  __device__ int jout_lo(int I) const { return max(0, h - I); }
  __device__ int jout_hi(int I) const { return min(Nt - 1, l - 1 - I); }
};

// Stage 1: M[I, J'] = sum_{I' in S1 column J', I' <= I} L^B[I, I'] E[I', J'].
__global__ void __launch_bounds__(256)
k_band1_simt(Band bd, const float* __restrict__ LB, int64_t ldb, const float* __restrict__ E,
             float* __restrict__ M, int64_t ldx) {
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
      As[r][c] = LB[((int64_t)I * TILE + r) * ldb + (int64_t)Ip * TILE + c];
      Bs[r][c] = E[((int64_t)Ip * TILE + r) * ldx + (int64_t)Jp * TILE + c];
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
  for (int u = 0; u < 4; ++u)
    M[((int64_t)I * TILE + tr) * ldx + (int64_t)Jp * TILE + tc + u] = acc[u];
}

// Stage 2: X[I, J] += sum_{J' in [max(0, k - I), min(J, h - 1)]} M[I, J'] L^A[J, J']^T.
__global__ void __launch_bounds__(256)
k_band2_simt(Band bd, const float* __restrict__ LA, int64_t lda, const float* __restrict__ M,
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
      As[r][c] = M[((int64_t)I * TILE + r) * ldx + (int64_t)Jp * TILE + c];
      Bs[c][r] = LA[((int64_t)J * TILE + r) * lda + (int64_t)Jp * TILE + c];
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
  float *X, *E, *M;
  const float *LA, *LB;
  const float *scales, *zeros;
  uint8_t* codes;
  int* status;
  cudaStream_t s;
};

static void leaf(const SolveArgs& a, int K) {
  const int ilo = max(0, K - (a.Nt - 1)), ihi = min(K, a.Mt - 1);
  LaunchScope ls(kFamLeaf, a.s);
  k_leaf<<<ihi - ilo + 1, 32, 0, a.s>>>(K, a.Mt, a.Nt, a.m, a.n, a.X, a.E, a.np, a.LB, a.mp,
                                        a.LA, a.np, a.scales, a.zeros, a.G, a.gsz, a.qmax,
                                        a.codes, a.status);
}

static void band(const SolveArgs& a, int k, int h, int l) {
  Band bd{k, h, l, a.Mt, a.Nt};
  dim3 g1(h, a.Mt), g2(l - h, a.Mt);
  {
    LaunchScope ls(kFamBand1, a.s);
    k_band1_simt<<<g1, 256, 0, a.s>>>(bd, a.LB, a.mp, a.E, a.M, a.np);
  }
  {
    LaunchScope ls(kFamBand2, a.s);
    k_band2_simt<<<g2, 256, 0, a.s>>>(bd, a.LA, a.np, a.M, a.X, a.np);
  }
}

static void rec(const SolveArgs& a, int k, int l) {
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
  a.E = (float*)(ws + sl.off_E);
  a.M = (float*)(ws + sl.off_M);
  a.LB = (const float*)(f + fl.off_LB);
  a.LA = (const float*)(f + fl.off_LA);
  a.scales = scales; a.zeros = zeros; a.codes = codes;
  a.status = (int*)(ws + sl.off_status);
  a.s = s;
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
  if (prerounding) {
    const int64_t tot = (int64_t)m * n;
    LaunchScope ls(kFamCopy, s);
    k_copy_out<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(a.X, a.np, m, n, prerounding);
  }
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}

}  // namespace bakron
