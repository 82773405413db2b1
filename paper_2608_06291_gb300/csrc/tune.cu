// Per-shape schedule thresholds and the autotuner that fills them
// (bakron_autotune, include/bakron.h).  The recursion itself is fixed by
// Alg. 5; what is tuned is only which kernels run each node, so every choice
// gives the same result up to fp32 summation order.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include <map>
#include <mutex>
#include <tuple>

#include "common.cuh"
#include "tune.cuh"
#include "solve.cuh"

namespace bakron {

namespace {
std::mutex g_mu;
std::map<std::tuple<int, int, int>, Tuning> g_table;   // (device, m, n) -> thresholds

int current_device() {
  int d = 0;
  return cudaGetDevice(&d) == cudaSuccess ? d : -1;
}

void env_override(const char* name, int& field) {
  const char* e = getenv(name);
  if (e && *e) field = atoi(e);
}
}  // namespace

Tuning tuning_for(int m, int n) {
  Tuning t = kDefaultTuning;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_table.find(std::make_tuple(current_device(), m, n));
    if (it != g_table.end()) t = it->second;
  }
  env_override("BAKRON_TC_MIN_BAND", t.tc_min_band);
  env_override("BAKRON_FUSED_MAX_BAND", t.fused_max_band);
  env_override("BAKRON_SUBTREE_MAX", t.subtree_max);
  env_override("BAKRON_LEAF_BLOCK", t.leaf_block);
  env_override("BAKRON_LEAF_FLOW", t.leaf_flow);
  return t;
}

}  // namespace bakron

using namespace bakron;

extern "C" {

int bakron_autotune(const void* W, int wdtype, int m, int n, int64_t ldw, const void* factors,
                    int bits, int group_size, uint8_t* codes, float* scales, float* zeros,
                    void* workspace, size_t workspace_bytes, int* tc_min_band,
                    int* fused_max_band, int* leaf_block, float* best_ms, void* stream) {
  if (!W || !factors || !codes || !scales || !zeros || !workspace || m < 1 || n < 1)
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || bits < 1 || bits > 8) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  if (workspace_bytes < bakron_workspace_bytes(m, n)) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  static const int kTc[] = {0, 4, 6, 8, 12, 16, 24};
  static const int kFused[] = {2, 4};
  static const int kBlock[] = {4, 8, 16};
  cudaEvent_t e0, e1;
  BK_CUDA_OK(cudaEventCreate(&e0));
  if (cudaEventCreate(&e1) != cudaSuccess) {
    cudaEventDestroy(e0);
    return BAKRON_ERR_CUDA;
  }
  Tuning best = kDefaultTuning;
  env_override("BAKRON_LEAF_FLOW", best.leaf_flow);   // not tuned: the default or the environment
  float best_t = -1.f;
  int rc = BAKRON_OK;
  for (int tc : kTc) {
    for (int fu : kFused) {
     for (int lb : kBlock) {
      const Tuning cand{tc, fu, 0, lb, best.leaf_flow};
      float t_min = -1.f;
      for (int rep = 0; rep < 3 && rc == BAKRON_OK; ++rep) {   // rep 0 warms up
        if (cudaEventRecord(e0, s) != cudaSuccess) { rc = BAKRON_ERR_CUDA; break; }
        rc = solve_impl(W, wdtype, m, n, ldw, factors, (1 << bits) - 1, group_size, codes,
                        scales, zeros, nullptr, workspace, s, &cand, false, false);
        if (rc != BAKRON_OK) break;
        if (cudaEventRecord(e1, s) != cudaSuccess) { rc = BAKRON_ERR_CUDA; break; }
        rc = bakron_read_status(workspace, stream);   // synchronises the stream
        if (rc != BAKRON_OK) break;
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, e0, e1) != cudaSuccess) { rc = BAKRON_ERR_CUDA; break; }
        if (rep > 0 && (t_min < 0.f || ms < t_min)) t_min = ms;
      }
      if (rc != BAKRON_OK) break;
      if (best_t < 0.f || t_min < best_t) {
        best_t = t_min;
        best = cand;
      }
     }
     if (rc != BAKRON_OK) break;
    }
    if (rc != BAKRON_OK) break;
  }
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (rc != BAKRON_OK) return rc;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    g_table[std::make_tuple(current_device(), m, n)] = best;
  }
  if (tc_min_band) *tc_min_band = best.tc_min_band;
  if (fused_max_band) *fused_max_band = best.fused_max_band;
  if (leaf_block) *leaf_block = best.leaf_block;
  if (best_ms) *best_ms = best_t;
  return BAKRON_OK;
}

int bakron_get_tuning(int m, int n, int* tc_min_band, int* fused_max_band, int* leaf_block) {
  if (m < 1 || n < 1) return BAKRON_ERR_INVALID_ARG;
  const Tuning t = tuning_for(m, n);
  if (tc_min_band) *tc_min_band = t.tc_min_band;
  if (fused_max_band) *fused_max_band = t.fused_max_band;
  if (leaf_block) *leaf_block = t.leaf_block;
  return BAKRON_OK;
}

void bakron_autotune_clear(void) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_table.clear();
}

}  // extern "C"
