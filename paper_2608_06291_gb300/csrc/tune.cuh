// Schedule thresholds of the solve (which Alg. 5 nodes run on which
// kernels): environment overrides, then a per-shape table filled by
// bakron_autotune, then defaults measured on GB300.  Host side only.
#pragma once

namespace bakron {

struct Tuning {
  int tc_min_band;     // nodes spanning >= this many tile anti-diagonals: tensor cores (<= 0: never)
  int fused_max_band;  // narrower CUDA-core nodes spanning <= this many: both stages in one launch
  int subtree_max;     // ranges spanning <= this many: one persistent cooperative launch (< 2: never)
  int leaf_block;      // ranges spanning <= this many: a block of leaves absorbing the nodes inside
  int leaf_flow;       // nonzero: a block of leaves is one dataflow launch (else one per anti-diagonal)
};

// Defaults: 4096 x 4096 solves are fastest with blocks of up to 8 leaves
// (no node narrower than 9 anti-diagonals is left) and tensor cores for
// every node above them.
constexpr Tuning kDefaultTuning{6, 2, 0, 8, 0};

// Thresholds for an m x n solve on the current device: the table entry if
// bakron_autotune stored one, else the defaults; each BAKRON_TC_MIN_BAND,
// BAKRON_FUSED_MAX_BAND, BAKRON_SUBTREE_MAX, BAKRON_LEAF_BLOCK that is set
// overrides its field.
Tuning tuning_for(int m, int n);

}  // namespace bakron
