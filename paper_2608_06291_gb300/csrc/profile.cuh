// Launch bracketing for the optional per-family timing (profile.cu).
#pragma once
#include <cuda_runtime.h>

namespace bakron {

enum {
  kFamInit = 0,
  kFamLeaf = 1,
  kFamBand1 = 2,    // SIMT band stage 1
  kFamBand2 = 3,    // SIMT band stage 2
  kFamCopy = 4,
  kFamTc1 = 5,      // tensor-core band stage 1
  kFamTc2 = 6,      // tensor-core band stage 2
  kFamFused = 7,    // both SIMT stages of a narrow node in one launch
  kFamSubtree = 8,  // persistent cooperative launch of a narrow range (leaves + bands)
  kFamilies = 9
};

// Counts one kernel launch; when profiling is on, records an event on the
// stream at construction and another at destruction (wrap exactly one launch).
class LaunchScope {
 public:
  // `flops`: algorithmic floating-point work of the launch (0 if not tracked)
  LaunchScope(int family, cudaStream_t s, double flops = 0.0);
  ~LaunchScope();
  LaunchScope(const LaunchScope&) = delete;
  LaunchScope& operator=(const LaunchScope&) = delete;

 private:
  int family_;
  cudaStream_t s_;
  void* a_;
  double flops_;
};

void reset_launch_count();
int launch_count();            // kernels enqueued on this host thread since the reset
void set_launch_count(int n);
bool profiling_on();

}  // namespace bakron
