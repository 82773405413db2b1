// Tensor-core (tcgen05, 3xTF32) band products: host interface (tc_gemm.cu).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace bakron {

// Device operands of the band products, in the solve's workspace/factor layout.
struct TcOperands {
  int64_t mp, np;      // padded sides (multiples of 128)
  int Mt, Nt;          // real 32-tiles per side
  const float *LBH, *LBL, *LAH, *LAL;
  float *EtH, *EtL, *MH, *ML, *X;
  int* status;
};

// TMA descriptors of every operand plane (built on the host per solve call).
struct TcMaps {
  CUtensorMap LB2, Et2, M2, LA2;   // hi/lo pairs in one box (32 columns x 128 rows x 2 planes)
  CUtensorMap Et2h, LA2h;          // the same in 64-row boxes: one half of B for CTA pairs
  CUtensorMap Eth, Etl;            // E^T planes in 32-row boxes (stage-1 sub-tiles at the band's edge)
  CUtensorMap Mh, Ml;              // M planes in 128-row boxes: stage-1 TMA store targets
  CUtensorMap X32;                 // X in 32 x 32 boxes: stage-2 TMA reduce-add target
};

bool tc_band_maps(TcMaps& maps, const TcOperands& op);

// Bound, in clock64 cycles, of every working device wait (BAKRON_SPIN_CYCLES,
// default about 2 s): a wait that runs out records BAKRON_ERR_TIMEOUT.
long long spin_cycles_from_env();

// Stage 1 (M = L^B E on the band [k, h)) or stage 2 (X += M L^A^T on the
// band [h, l)) of one Alg. 5 node, over 128 x 128 output blocks.
// `stamp`: the launch's timeline stamp slot (null: none).
int tc_band_stage(int stage, const TcMaps& maps, const TcOperands& op, int k, int h, int l,
                  cudaStream_t s, unsigned long long* stamp = nullptr);

// Stage `stage` of node (k, h, l) for H <= 32 problems of one shape (op gives
// the shape; maps[p] and status[p] are problem p's) in one launch.
int tc_band_stage_heads(int stage, int H, const TcMaps* const* maps, int* const* status,
                        const TcOperands& op, int k, int h, int l, cudaStream_t s,
                        unsigned long long* stamp = nullptr);

// The column-band update of the B = I (GPTQ) schedule over 128 x 128 output
// blocks: X[:, S2] += E[:, S1] L^A[S2, S1]^T, S1 = tile columns [k, h), S2 =
// [h, l), with E in the M planes (row-major hi/lo).
int tc_cols_stage(const TcMaps& maps, const TcOperands& op, int k, int h, int l, cudaStream_t s,
                  unsigned long long* stamp = nullptr);

}  // namespace bakron
