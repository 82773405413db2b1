// bakron_prepare: damping and unit-lower factors of the Kronecker Grams.
//
// Paper: Alg. 2, first two lines (L = Cholesky(H^-1), columns scaled to a unit
// diagonal), done once at top level (Appendix, equivalence proof, conventions);
// damping H + damp * mean(diag H) * I (Sec. 4, Appendix "Experiments").
//
// Route.  With R = RevCholesky(H_d) (R^T R = H_d, R lower), Cholesky(H_d^-1) =
// R^-1, so the unit-lower factor is R^-1 diag(R).  R comes from the ordinary
// Cholesky of the reversed matrix: J H_d J = C C^T gives R = J C^T J, hence
//     Lhat[i][j] = (C^-1)[d-1-j][d-1-i] * C[d-1-j][d-1-j]     (i >= j).
// So: reverse+damp -> blocked Cholesky of C -> blocked inverse of C -> flip,
// transpose and scale into the fp32 factor buffer.  No explicit H^-1.
//
// Precision.  The factorisation runs in fp64 and is rounded to fp32 once at
// the end.  An fp32 factorisation has relative error ~kappa * 2^-24 (1e-5 at
// the condition numbers of the power-law Grams); error feedback multiplies
// that into the pre-rounding values by the factor's column sums, which leaves
// it too close to the 1e-4 grid-unit tie band on 4096-wide problems.  fp32 is
// kept as an option (BAKRON_PREPARE_FP32=1) for speed.
#include <cuda_runtime.h>
#include <math.h>
#include <stdlib.h>

#include "common.cuh"

namespace bakron {

constexpr int NB = 64;          // Cholesky / inverse block size
constexpr int GT = 64;          // SIMT GEMM output tile
constexpr int GK = 16;          // SIMT GEMM k-chunk

// ---------------------------------------------------------------- damping
template <typename RT>
__global__ void k_diag_sum(const float* A, int d, RT* out) {
  RT acc = 0;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < d; i += gridDim.x * blockDim.x)
    acc += (RT)A[(int64_t)i * d + i];
  for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) atomicAdd(out, acc);
}

// C[i][j] = A_d[d-1-j][d-1-i] for i >= j (reads the lower triangle of A);
// C[i][j] = 0 above the diagonal.  Padding rows/cols (>= d) are the identity.
template <typename RT>
__global__ void k_reverse_damp(const float* A, int d, int64_t dp, float damp,
                               const RT* diag_sum, RT* C) {
  int64_t i = blockIdx.y * (int64_t)blockDim.y + threadIdx.y;
  int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= dp || j >= dp) return;
  RT v = 0;
  if (i < d && j < d) {
    if (j <= i) {
      v = (RT)A[(int64_t)(d - 1 - j) * d + (d - 1 - i)];
      if (i == j) v += (RT)damp * (*diag_sum / (RT)d);
    }
  } else if (i == j) {
    v = 1;
  }
  C[i * dp + j] = v;
}

// ------------------------------------------------- diagonal block Cholesky
// Factor the b x b block at (k0, k0) in place (lower) and write its inverse
// into Dinv (NB x NB, row-major).  A non-positive pivot raises NOT_SPD and is
// replaced by 1 so that no NaN spreads.
template <typename RT>
__global__ void k_potrf_block(RT* C, int64_t ldc, int k0, int b, RT* Dinv, int* status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  RT (*s)[NB + 1] = reinterpret_cast<RT (*)[NB + 1]>(smem_raw);
  RT (*inv)[NB + 1] = reinterpret_cast<RT (*)[NB + 1]>(smem_raw + sizeof(RT) * NB * (NB + 1));
  const int t = threadIdx.x, nt = blockDim.x;
  for (int e = t; e < NB * NB; e += nt) {
    int r = e / NB, c = e % NB;
    s[r][c] = (r < b && c <= r) ? C[(int64_t)(k0 + r) * ldc + k0 + c] : (r == c ? RT(1) : RT(0));
    inv[r][c] = 0;
  }
  __syncthreads();
  for (int j = 0; j < b; ++j) {
    if (t == 0) {
      RT p = s[j][j];
      if (!(p > 0)) { raise_status(status, BAKRON_ERR_NOT_SPD); p = 1; }
      s[j][j] = sqrt(p);
    }
    __syncthreads();
    RT piv = s[j][j];
    for (int r = j + 1 + t; r < b; r += nt) s[r][j] /= piv;
    __syncthreads();
    // trailing update of the lower part of columns j+1..b-1
    for (int e = t; e < (b - j - 1) * (b - j - 1); e += nt) {
      int r = j + 1 + e / (b - j - 1), c = j + 1 + e % (b - j - 1);
      if (c <= r) s[r][c] -= s[r][j] * s[c][j];
    }
    __syncthreads();
  }
  // inverse of the lower-triangular block, right-looking: row k of the
  // inverse is final once divided by the pivot, then every later row r drops
  // s[r][k] times it (independent updates spread over the whole CTA instead
  // of one dependent chain per column)
  for (int e = t; e < NB * NB; e += nt) {
    const int r = e / NB, c = e % NB;
    inv[r][c] = (r == c) ? RT(1) : RT(0);
  }
  __syncthreads();
  for (int k = 0; k < NB; ++k) {
    for (int c = t; c <= k; c += nt) inv[k][c] /= s[k][k];
    __syncthreads();
    const int w = k + 1, rows = NB - 1 - k;
    for (int e = t; e < rows * w; e += nt) {
      const int r = k + 1 + e / w, c = e % w;
      inv[r][c] -= s[r][k] * inv[k][c];
    }
    __syncthreads();
  }
  for (int e = t; e < NB * NB; e += nt) {
    int r = e / NB, c = e % NB;
    if (r < b && c <= r) C[(int64_t)(k0 + r) * ldc + k0 + c] = s[r][c];
    Dinv[e] = inv[r][c];
  }
}

// ------------------------------------------------------------ SIMT GEMM
// C[M x N] = beta*C + alpha * op(A) * op(B):  op(A) = A (M x K) or A^T (A
// given K x M), op(B) = B (K x N) or B^T (B given N x K).  64 x 64 output
// tiles, 256 threads, 4 x 4 per thread; each operand is staged with the
// thread index running along its contiguous dimension.
// mode bit 1: only tiles with tile_row >= tile_col (lower part, for SYRK).
// mode bit 2: op(B) is lower triangular: skip k < tile_col * 64.
// mode bit 4: op(A) is upper triangular: skip k < tile_row * 64.
// mode bit 8: op(A) is lower triangular: skip k >= (tile_row + 1) * 64.
// Each CTA reads all of its A rows before writing, so C may alias A when
// N <= 64 (the panel solve uses this).
enum { GM_LOWER_C = 1, GM_TRI_B = 2, GM_UPPER_A = 4, GM_LOWER_A = 8 };

template <typename RT, bool TRANS_A, bool TRANS_B>
__global__ void __launch_bounds__(256) k_gemm(int M, int N, int K, RT alpha,
                                              const RT* A, int64_t lda,
                                              const RT* B, int64_t ldb, RT beta,
                                              RT* C, int64_t ldc, int mode) {
  const int tr = blockIdx.y, tc = blockIdx.x;
  if ((mode & GM_LOWER_C) && tc > tr) return;
  __shared__ RT As[GK][GT + 1];
  __shared__ RT Bs[GK][GT + 1];
  const int t = threadIdx.x;
  const int ty = t / 16, tx = t % 16;
  RT acc[4][4] = {};
  int kbeg = 0, kend = K;
  if (mode & GM_TRI_B) kbeg = max(kbeg, tc * GT);
  if (mode & GM_UPPER_A) kbeg = max(kbeg, tr * GT);
  if (mode & GM_LOWER_A) kend = min(kend, (tr + 1) * GT);
  for (int k0 = kbeg; k0 < kend; k0 += GK) {
    for (int e = t; e < GK * GT; e += 256) {
      const int kk = TRANS_A ? e / GT : e % GK, r = TRANS_A ? e % GT : e / GK;
      const int gr = tr * GT + r, gk = k0 + kk;
      As[kk][r] = (gr < M && gk < K) ? (TRANS_A ? A[(int64_t)gk * lda + gr]
                                                : A[(int64_t)gr * lda + gk])
                                     : RT(0);
    }
    for (int e = t; e < GK * GT; e += 256) {
      const int kk = TRANS_B ? e % GK : e / GT, c = TRANS_B ? e / GK : e % GT;
      const int gc = tc * GT + c, gk = k0 + kk;
      Bs[kk][c] = (gc < N && gk < K) ? (TRANS_B ? B[(int64_t)gc * ldb + gk]
                                                : B[(int64_t)gk * ldb + gc])
                                     : RT(0);
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GK; ++kk) {
      RT a[4], bb[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bb[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] += a[i] * bb[j];
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int gr = tr * GT + ty * 4 + i, gc = tc * GT + tx * 4 + j;
      if (gr < M && gc < N) {
        if ((mode & GM_LOWER_C) && gc > gr) continue;
        RT* p = C + (int64_t)gr * ldc + gc;
        *p = (beta == RT(0) ? RT(0) : beta * *p) + alpha * acc[i][j];
      }
    }
}

template <typename RT>
static void gemm(cudaStream_t s, int M, int N, int K, RT alpha, const RT* A, int64_t lda,
                 bool transA, const RT* B, int64_t ldb, bool transB, RT beta, RT* C, int64_t ldc,
                 int mode) {
  if (M <= 0 || N <= 0) return;
  dim3 grid(ceil_div(N, GT), ceil_div(M, GT));
  if (transA && transB)
    k_gemm<RT, true, true><<<grid, 256, 0, s>>>(M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, mode);
  else if (transB)
    k_gemm<RT, false, true><<<grid, 256, 0, s>>>(M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, mode);
  else if (transA)
    k_gemm<RT, true, false><<<grid, 256, 0, s>>>(M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, mode);
  else
    k_gemm<RT, false, false><<<grid, 256, 0, s>>>(M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, mode);
}

// Copy a b x b block of Dinv into X's diagonal block (lower part only).
template <typename RT>
__global__ void k_put_diag(const RT* Dinv, int b, RT* X, int64_t ldx, int i0) {
  int r = blockIdx.x, c = threadIdx.x;
  if (r < b && c < b) X[(int64_t)(i0 + r) * ldx + i0 + c] = (c <= r) ? Dinv[r * NB + c] : RT(0);
}

// Lhat[i][j] = Xinv[d-1-j][d-1-i] * C[d-1-j][d-1-j]  (i > j), 1 on the
// diagonal, 0 above, identity on the padding; rdiag[i] = C[d-1-i][d-1-i].
template <typename RT>
__global__ void k_assemble(const RT* C, const RT* Xinv, int64_t dp, int d, float* L,
                           float* Llo, int64_t ldl, int64_t Lp, float* rdiag) {
  __shared__ float tile[32][33];
  const int bx = blockIdx.x * 32, by = blockIdx.y * 32;
  // read transposed source block: source row a = d-1-j, col b = d-1-i
  for (int yy = threadIdx.y; yy < 32; yy += blockDim.y) {
    int j = bx + yy;          // destination column
    int i = by + threadIdx.x; // destination row
    float v = 0.f;
    if (i < d && j < d && i > j) {
      int64_t a = d - 1 - j, bcol = d - 1 - i;
      v = (float)(Xinv[a * dp + bcol] * C[a * dp + a]);
    }
    tile[yy][threadIdx.x] = v;
  }
  __syncthreads();
  for (int yy = threadIdx.y; yy < 32; yy += blockDim.y) {
    int i = by + yy, j = bx + threadIdx.x;
    if (i < Lp && j < Lp) {
      float v = tile[threadIdx.x][yy];
      if (i == j) v = 1.f;
      else if (i >= d || j >= d) v = 0.f;
      const float hi = tf32_hi(v);
      L[(int64_t)i * ldl + j] = hi;
      Llo[(int64_t)i * ldl + j] = v - hi;
    }
  }
  if (blockIdx.x == 0 && threadIdx.y == 0) {
    int i = by + threadIdx.x;
    if (i < Lp) rdiag[i] = (i < d) ? (float)C[(int64_t)(d - 1 - i) * dp + (d - 1 - i)] : 1.f;
  }
}

// X[i0 .. i0 + n) x [i0 .. i0 + n) = inverse of the lower triangle of C's
// diagonal block there, by recursive halving at a multiple of NB: with
// C = [[C11, 0], [C21, C22]], X11 = C11^-1 and X22 = C22^-1 (recursively; a
// block of at most NB is the inverse the panel factorisation left in Dinv),
// X21 = -X22 (C21 X11).  The product C21 X11 is kept transposed in C's upper
// triangle above the node's diagonal block (C11's rows, C22's columns),
// which the lower Cholesky factor leaves unused; X above the diagonal stays
// as zeroed.  Every level is two GEMMs over whole halves, so the work runs
// on the whole GPU (a block-row recurrence gives each step at most i0 / 64
// output tiles).
template <typename RT>
static void inv_lower(cudaStream_t s, RT* C, RT* X, int64_t dp, const RT* Dinv, int i0, int n) {
  if (n <= NB) {
    k_put_diag<RT><<<n, NB, 0, s>>>(Dinv + (int64_t)(i0 / NB) * NB * NB, n, X, dp, i0);
    return;
  }
  const int n1 = (ceil_div(n, NB) / 2) * NB, n2 = n - n1;
  inv_lower<RT>(s, C, X, dp, Dinv, i0, n1);
  inv_lower<RT>(s, C, X, dp, Dinv, i0 + n1, n2);
  RT* R = C + (int64_t)i0 * dp + (i0 + n1);                    // n1 x n2, above the diagonal
  const RT* C21 = C + (int64_t)(i0 + n1) * dp + i0;            // n2 x n1
  const RT* X11 = X + (int64_t)i0 * dp + i0;                   // n1 x n1, lower
  const RT* X22 = X + (int64_t)(i0 + n1) * dp + (i0 + n1);     // n2 x n2, lower
  RT* X21 = X + (int64_t)(i0 + n1) * dp + i0;                  // n2 x n1
  // R = (C21 X11)^T = X11^T C21^T  (X11^T upper triangular)
  gemm<RT>(s, n1, n2, n1, RT(1), X11, dp, true, C21, dp, true, RT(0), R, dp, GM_UPPER_A);
  // X21 = -X22 R^T  (X22 lower triangular)
  gemm<RT>(s, n2, n1, n2, RT(-1), X22, dp, false, R, dp, true, RT(0), X21, dp, GM_LOWER_A);
}

// One Gram -> one unit-lower factor (fp32, Lp x Lp) and its RevCholesky diagonal.
template <typename RT>
static int factor_one(const float* H, int d, float damp, float* L, float* Llo, int64_t Lp,
                      float* rdiag, void* workspace, const PrepareLayout& lay, cudaStream_t s) {
  char* ws = (char*)workspace;
  int* status = (int*)(ws + lay.off_status);
  const int64_t dp = round_up(d, PAD);
  RT* C = (RT*)(ws + lay.off_C);        // dp x dp: reversed damped Gram -> its Cholesky factor
  RT* X = (RT*)(ws + lay.off_Linv);     // dp x dp: inverse of that factor
  RT* Dinv = (RT*)(ws + lay.off_T);     // inverses of the NB x NB diagonal blocks
  RT* sum = (RT*)(ws + lay.off_scalar);
  const size_t smem = 2 * sizeof(RT) * NB * (NB + 1);
  BK_CUDA_OK(cudaFuncSetAttribute(k_potrf_block<RT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)smem));
  BK_CUDA_OK(cudaMemsetAsync(sum, 0, sizeof(RT), s));
  BK_CUDA_OK(cudaMemsetAsync(X, 0, sizeof(RT) * dp * dp, s));
  int nblk = ceil_div(d, 256);
  k_diag_sum<RT><<<nblk > 64 ? 64 : nblk, 256, 0, s>>>(H, d, sum);
  {
    dim3 blk(32, 8), grid(ceil_div((int)dp, 32), ceil_div((int)dp, 8));
    k_reverse_damp<RT><<<grid, blk, 0, s>>>(H, d, dp, damp, sum, C);
  }
  // right-looking blocked Cholesky of C (lower, in place)
  for (int k0 = 0; k0 < d; k0 += NB) {
    const int b = d - k0 < NB ? d - k0 : NB;
    RT* Dk = Dinv + (int64_t)(k0 / NB) * NB * NB;
    k_potrf_block<RT><<<1, 256, smem, s>>>(C, dp, k0, b, Dk, status);
    const int rest = d - k0 - b;
    if (rest > 0) {
      RT* P = C + (int64_t)(k0 + b) * dp + k0;
      // panel solve P <- P L_kk^-T  (in place: one CTA per 64 whole rows, N = b <= 64)
      gemm<RT>(s, rest, b, b, RT(1), P, dp, false, Dk, NB, true, RT(0), P, dp, 0);
      // trailing update C22 -= P P^T on the lower tiles
      RT* C22 = C + (int64_t)(k0 + b) * dp + (k0 + b);
      gemm<RT>(s, rest, rest, b, RT(-1), P, dp, false, P, dp, true, RT(1), C22, dp, GM_LOWER_C);
    }
  }
  // X = C^-1 by recursive halving (inv_lower)
  inv_lower<RT>(s, C, X, dp, Dinv, 0, d);
  {
    dim3 blk(32, 8), grid((unsigned)(Lp / 32), (unsigned)(Lp / 32));
    k_assemble<RT><<<grid, blk, 0, s>>>(C, X, dp, d, L, Llo, Lp, Lp, rdiag);
  }
  BK_CUDA_OK(cudaGetLastError());
  return BAKRON_OK;
}

int prepare_impl(const float* A, const float* B, int m, int n, float damp, void* factors,
                 void* workspace, cudaStream_t s) {
  FactorLayout fl(m, n);
  PrepareLayout pl(m, n);
  char* f = (char*)factors;
  const char* env = getenv("BAKRON_PREPARE_FP32");
  const bool fp32 = env && env[0] == '1';
  BK_CUDA_OK(cudaMemsetAsync((char*)workspace + pl.off_status, 0, 256, s));
  int rc;
  if (fp32) {
    rc = factor_one<float>(A, n, damp, (float*)(f + fl.off_LAH), (float*)(f + fl.off_LAL),
                           fl.np, (float*)(f + fl.off_rA), workspace, pl, s);
    if (rc == BAKRON_OK)
      rc = factor_one<float>(B, m, damp, (float*)(f + fl.off_LBH), (float*)(f + fl.off_LBL),
                             fl.mp, (float*)(f + fl.off_rB), workspace, pl, s);
  } else {
    rc = factor_one<double>(A, n, damp, (float*)(f + fl.off_LAH), (float*)(f + fl.off_LAL),
                            fl.np, (float*)(f + fl.off_rA), workspace, pl, s);
    if (rc == BAKRON_OK)
      rc = factor_one<double>(B, m, damp, (float*)(f + fl.off_LBH), (float*)(f + fl.off_LBL),
                              fl.mp, (float*)(f + fl.off_rB), workspace, pl, s);
  }
  if (rc == BAKRON_OK) rc = build_leaf_blocks(fl, f, s);
  return rc;
}

}  // namespace bakron
