// Optional per-kernel-family timing of bakron_solve (for benchmarks), and the
// launch counter.  Host-side only.
//
// Two modes.  Event mode brackets each launch with CUDA events; the events
// serialise the launches (a kernel can no longer start its prologue while the
// previous one runs), so its times add up to more than the solve takes.
// Timeline mode has every launch stamp, on the device, when its CTAs start
// their dependent work and when the last one ends (global nanosecond timer);
// the solve's launch sequence is recorded once (typically while a CUDA graph
// of the solve is captured) and each replay's stamps are turned into a
// partition of that replay's time: launch i owns the interval from the end of
// launch i - 1 to its own end (launch 0 from its start).  The family times
// then add up to the replay's device time.
#include <cuda_runtime.h>

#include <algorithm>
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
constexpr int kMaxSlots = 1 << 15;   // launches of one solve in timeline mode

std::mutex g_mu;
int g_mode = 0;                      // 0 off, 1 events, 2 timeline
std::vector<Pending> g_pending;
std::vector<cudaEvent_t> g_free;
int g_launches[kFamilies] = {};
double g_ms[kFamilies] = {};
double g_flops[kFamilies] = {};
double g_timeline_ms = 0.0;          // sum over collected replays of (last end - first start)
int g_replays = 0;
unsigned long long* g_stamps = nullptr;   // device, 2 per slot
std::vector<std::pair<int, double>> g_slots;   // (family, flops) of the recorded solve
std::vector<unsigned long long> g_last;         // stamps of the last collected run
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

// starts at the largest value (atomicMin), ends at zero (atomicMax)
__global__ void k_clear_stamps(unsigned long long* st, int words) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < words) st[i] = (i & 1) ? 0ull : ~0ull;
}
cudaError_t clear_stamps(cudaStream_t s) {
  const int words = 2 * kMaxSlots;
  k_clear_stamps<<<(words + 255) / 256, 256, 0, s>>>(g_stamps, words);
  return cudaGetLastError();
}
}  // namespace

LaunchScope::LaunchScope(int family, cudaStream_t s, double flops)
    : family_(family), s_(s), a_(nullptr), flops_(flops), stamp_(nullptr) {
  ++t_launch_count;
  if (g_mode == 0) return;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_mode == 2) {
    if ((int)g_slots.size() < kMaxSlots) {
      stamp_ = g_stamps + 2 * g_slots.size();
      g_slots.push_back({family, flops});
    }
    return;
  }
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

void reset_launch_count() {
  t_launch_count = 0;
  if (g_mode == 2) {
    std::lock_guard<std::mutex> lk(g_mu);
    g_slots.clear();
  }
}
int launch_count() { return t_launch_count; }
void set_launch_count(int n) { t_launch_count = n; }

bool profiling_on() { return g_mode != 0; }

}  // namespace bakron

using namespace bakron;

extern "C" int bakron_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_mu);
  drain_locked();
  for (int f = 0; f < kFamilies; ++f) { g_launches[f] = 0; g_ms[f] = 0.0; g_flops[f] = 0.0; }
  g_timeline_ms = 0.0;
  g_replays = 0;
  g_slots.clear();
  if (on == 2) {
    if (!g_stamps &&
        cudaMalloc(&g_stamps, sizeof(unsigned long long) * 2 * kMaxSlots) != cudaSuccess) {
      g_stamps = nullptr;
      g_mode = 0;
      return BAKRON_ERR_CUDA;
    }
    if (clear_stamps(0) != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) {
      g_mode = 0;
      return BAKRON_ERR_CUDA;
    }
  }
  g_mode = on == 2 ? 2 : (on ? 1 : 0);
  return BAKRON_OK;
}

extern "C" int bakron_profile_collect(void* stream) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_mode != 2) return BAKRON_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  const size_t n = g_slots.size();
  std::vector<unsigned long long> h(2 * std::max<size_t>(n, 1));
  BK_CUDA_OK(cudaStreamSynchronize(s));
  if (n) BK_CUDA_OK(cudaMemcpy(h.data(), g_stamps, sizeof(unsigned long long) * 2 * n,
                               cudaMemcpyDeviceToHost));
  g_last.assign(h.begin(), h.begin() + 2 * n);
  // launches in enqueue order; a launch without stamps (its kernel takes no
  // stamp slot, or none of its CTAs had work) owns no time
  unsigned long long first = 0, prev_end = 0;
  bool any = false;
  for (size_t i = 0; i < n; ++i) {
    const unsigned long long b = h[2 * i], e = h[2 * i + 1];
    const int fam = g_slots[i].first;
    g_launches[fam] += 1;
    g_flops[fam] += g_slots[i].second;
    if (e == 0) continue;
    if (!any) {
      first = b <= e ? b : e;
      prev_end = first;
      any = true;
    }
    if (e > prev_end) {
      g_ms[fam] += 1e-6 * (double)(e - prev_end);
      prev_end = e;
    }
  }
  if (any) g_timeline_ms += 1e-6 * (double)(prev_end - first);
  ++g_replays;
  BK_CUDA_OK(clear_stamps(s));
  BK_CUDA_OK(cudaStreamSynchronize(s));
  return BAKRON_OK;
}

extern "C" int bakron_profile_read(int family, int* launches, double* ms, double* flops) {
  if (family < -1 || family >= kFamilies || !launches || !ms) return BAKRON_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  drain_locked();
  if (family == -1) {   // timeline mode: collected replays and their summed span
    *launches = g_replays;
    *ms = g_timeline_ms;
    if (flops) *flops = 0.0;
    return BAKRON_OK;
  }
  *launches = g_launches[family];
  *ms = g_ms[family];
  if (flops) *flops = g_flops[family];
  return BAKRON_OK;
}

extern "C" int bakron_last_launches(void) { return t_launch_count; }

extern "C" int bakron_profile_launch_stamps(int max, int* family, double* flops,
                                            double* start_us, double* end_us) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (max < 0 || !family || !flops || !start_us || !end_us) return -BAKRON_ERR_INVALID_ARG;
  const size_t n = std::min(g_slots.size(), g_last.size() / 2);
  unsigned long long t0 = ~0ull;
  for (size_t i = 0; i < n; ++i)
    if (g_last[2 * i + 1] != 0) t0 = std::min(t0, g_last[2 * i]);
  const int k = (int)std::min<size_t>(n, (size_t)max);
  for (int i = 0; i < k; ++i) {
    family[i] = g_slots[i].first;
    flops[i] = g_slots[i].second;
    const unsigned long long b = g_last[2 * i], e = g_last[2 * i + 1];
    start_us[i] = e ? 1e-3 * (double)(b - t0) : -1.0;
    end_us[i] = e ? 1e-3 * (double)(e - t0) : -1.0;
  }
  return (int)n;
}
