// Launch bracketing for the optional per-family timing (profile.cu).
#pragma once
#include <cuda_runtime.h>

namespace bakron {

enum { kFamInit = 0, kFamLeaf = 1, kFamBand1 = 2, kFamBand2 = 3, kFamCopy = 4, kFamilies = 5 };

// Counts one kernel launch; when profiling is on, records an event on the
// stream at construction and another at destruction (wrap exactly one launch).
class LaunchScope {
 public:
  LaunchScope(int family, cudaStream_t s);
  ~LaunchScope();
  LaunchScope(const LaunchScope&) = delete;
  LaunchScope& operator=(const LaunchScope&) = delete;

 private:
  int family_;
  cudaStream_t s_;
  void* a_;
};

void reset_launch_count();

}  // namespace bakron
