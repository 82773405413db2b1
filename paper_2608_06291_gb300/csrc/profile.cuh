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

// Counts one kernel launch.  Event mode (bakron_profile_enable(1)): records
// an event on the stream at construction and another at destruction (wrap
// exactly one launch).  Timeline mode (bakron_profile_enable(2)): takes the
// next stamp slot of the current solve, which the launch passes to its kernel
// (stamp(); null in the other modes).
class LaunchScope {
 public:
  // `flops`: algorithmic floating-point work of the launch (0 if not tracked)
  LaunchScope(int family, cudaStream_t s, double flops = 0.0);
  ~LaunchScope();
  LaunchScope(const LaunchScope&) = delete;
  LaunchScope& operator=(const LaunchScope&) = delete;
  unsigned long long* stamp() const { return stamp_; }

 private:
  int family_;
  cudaStream_t s_;
  void* a_;
  double flops_;
  unsigned long long* stamp_;
};

void reset_launch_count();    // also starts a new solve's stamp slots
int launch_count();            // kernels enqueued on this host thread since the reset
void set_launch_count(int n);
bool profiling_on();

}  // namespace bakron
