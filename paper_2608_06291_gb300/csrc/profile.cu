// Optional per-kernel-family timing of bakron_solve with CUDA events (for
// benchmarks), and the launch counter.  Host-side only.
#include <cuda_runtime.h>

#include <mutex>
#include <vector>

#include "common.cuh"
#include "profile.cuh"

namespace bakron {

namespace {
struct Pending {
  int family;
  cudaEvent_t a, b;
  double flops;
};
std::mutex g_mu;
bool g_on = false;
std::vector<Pending> g_pending;
std::vector<cudaEvent_t> g_free;
int g_launches[kFamilies] = {};
double g_ms[kFamilies] = {};
double g_flops[kFamilies] = {};
thread_local int t_launch_count = 0;

cudaEvent_t take_event() {
  if (!g_free.empty()) {
    cudaEvent_t e = g_free.back();
    g_free.pop_back();
    return e;
  }
  cudaEvent_t e;
  cudaEventCreate(&e);
  return e;
}

void drain_locked() {
  for (auto& p : g_pending) {
    float ms = 0.f;
    cudaEventSynchronize(p.b);
    cudaEventElapsedTime(&ms, p.a, p.b);
    g_ms[p.family] += ms;
    g_flops[p.family] += p.flops;
    g_launches[p.family] += 1;
    g_free.push_back(p.a);
    g_free.push_back(p.b);
  }
  g_pending.clear();
}
}  // namespace

LaunchScope::LaunchScope(int family, cudaStream_t s, double flops)
    : family_(family), s_(s), a_(nullptr), flops_(flops) {
  ++t_launch_count;
  if (!g_on) return;
  std::lock_guard<std::mutex> lk(g_mu);
  a_ = take_event();
  cudaEventRecord((cudaEvent_t)a_, s_);
}

LaunchScope::~LaunchScope() {
  if (!a_) return;
  std::lock_guard<std::mutex> lk(g_mu);
  cudaEvent_t b = take_event();
  cudaEventRecord(b, s_);
  g_pending.push_back({family_, (cudaEvent_t)a_, b, flops_});
}

void reset_launch_count() { t_launch_count = 0; }
int launch_count() { return t_launch_count; }
void set_launch_count(int n) { t_launch_count = n; }

bool profiling_on() { return g_on; }

}  // namespace bakron

using namespace bakron;

extern "C" int bakron_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_mu);
  drain_locked();
  for (int f = 0; f < kFamilies; ++f) { g_launches[f] = 0; g_ms[f] = 0.0; g_flops[f] = 0.0; }
  g_on = on != 0;
  return BAKRON_OK;
}

extern "C" int bakron_profile_read(int family, int* launches, double* ms, double* flops) {
  if (family < 0 || family >= kFamilies || !launches || !ms) return BAKRON_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  drain_locked();
  *launches = g_launches[family];
  *ms = g_ms[family];
  if (flops) *flops = g_flops[family];
  return BAKRON_OK;
}

extern "C" int bakron_last_launches(void) { return t_launch_count; }
