// Schedule thresholds of the solve (which Alg. 5 nodes run on which
// kernels): environment overrides, then a per-shape table filled by
// bakron_autotune, then defaults measured on GB300.  Host side only.
#pragma once

namespace bakron {

struct Tuning {
  int tc_min_band;     // nodes spanning >= this many tile anti-diagonals: tensor cores (<= 0: never)
  int fused_max_band;  // narrower CUDA-core nodes spanning <= this many: both stages in one launch
  int subtree_max;     // ranges spanning <= this many: one persistent cooperative launch (< 2: never)
};

// Defaults: 4096 x 4096 and 11008 x 4096 solves are fastest with tensor
// cores from 6 anti-diagonals up and no fused launches (a width-2 node is
// applied by its second leaf, so fused_max_band = 2 fuses nothing).
constexpr Tuning kDefaultTuning{6, 2, 0};

// Thresholds for an m x n solve on the current device: the table entry if
// bakron_autotune stored one, else the defaults; each BAKRON_TC_MIN_BAND,
// BAKRON_FUSED_MAX_BAND, BAKRON_SUBTREE_MAX that is set overrides its field.
Tuning tuning_for(int m, int n);

}  // namespace bakron
