// bakron_solve_batched: many independent solves of one shape in one call --
// the per-head problems of BoA-style attention Hessians (a block-diagonal
// output-side factor: one small B per head, a shared input-side A), which
// the paper names as the setting its local attention Hessians come from
// (Sec. 4, local Hessians; the BoA comparison).
//
// A small problem (e.g. 128 x 4096: 4 x 128 tiles) keeps only a few SMs busy
// at each step of its wavefront, so the problems run side by side: problem h
// is enqueued on lane h mod S of S library-owned streams, which fork from the
// caller's stream through an event and join back into it through one event
// per lane.  With one lane per problem (S = H), the leaves of all problems
// share one launch per tile anti-diagonal on the caller's stream, and so do
// the tensor-core band stages (one launch per stage, blockIdx.z = problem);
// only CUDA-core band products of narrow nodes run per problem on the lanes
// (solve_heads_impl).  Each lane owns one slice of the workspace and runs its problems
// one after another; a problem's kernels are those of bakron_solve (same
// schedule table, same programmatic dependent launch within its lane).  The
// fork/join is made of event records and waits only, so the whole call can
// be captured into a CUDA graph once the lane streams exist.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>
#include <vector>

#include "common.cuh"
#include "profile.cuh"
#include "tune.cuh"
#include "solve.cuh"

namespace bakron {

namespace {

constexpr int MAX_LANES = 32;

struct Lanes {
  cudaStream_t stream[MAX_LANES] = {};
  cudaEvent_t done[MAX_LANES] = {};
  cudaEvent_t fork = nullptr;
  int created = 0;
};

std::mutex g_lanes_mu;
std::vector<Lanes> g_lanes;   // per device

size_t slice_bytes(int m, int n) { return (size_t)round_up((int64_t)SolveLayout(m, n).bytes, 256); }

// Lanes 0..S-1 of the current device, created on first use (not while a
// stream capture is in progress: make the first call outside any capture).
int lanes_for(int S, Lanes** out) {
  int dev = 0;
  BK_CUDA_OK(cudaGetDevice(&dev));
  if ((int)g_lanes.size() <= dev) g_lanes.resize(dev + 1);
  Lanes& L = g_lanes[dev];
  if (!L.fork) BK_CUDA_OK(cudaEventCreateWithFlags(&L.fork, cudaEventDisableTiming));
  while (L.created < S) {
    const int i = L.created;
    BK_CUDA_OK(cudaStreamCreateWithFlags(&L.stream[i], cudaStreamNonBlocking));
    BK_CUDA_OK(cudaEventCreateWithFlags(&L.done[i], cudaEventDisableTiming));
    L.created = i + 1;
  }
  *out = &L;
  return BAKRON_OK;
}

}  // namespace
}  // namespace bakron

using namespace bakron;

extern "C" {

size_t bakron_batched_workspace_bytes(int m, int n, int streams) {
  if (m < 1 || n < 1 || streams < 1 || streams > MAX_LANES) return 0;
  const size_t one = bakron_workspace_bytes(m, n);
  if (one == 0) return 0;
  return (size_t)streams * slice_bytes(m, n);
}

int bakron_solve_batched(int H, const void* const* W, int wdtype, int m, int n, int64_t ldw,
                         const void* const* factors, int bits, int group_size,
                         uint8_t* const* codes, float* const* scales, float* const* zeros,
                         void* workspace, size_t workspace_bytes, int streams, int sync,
                         void* stream) {
  if (H < 1 || !W || !factors || !codes || !scales || !zeros || !workspace)
    return BAKRON_ERR_INVALID_ARG;
  if (streams < 1 || streams > MAX_LANES || bakron_workspace_bytes(m, n) == 0)
    return BAKRON_ERR_INVALID_ARG;
  if (wdtype != BAKRON_F32 && wdtype != BAKRON_BF16) return BAKRON_ERR_INVALID_ARG;
  if (ldw < n || bits < 1 || bits > 8) return BAKRON_ERR_INVALID_ARG;
  if (group_size < 0 || (group_size > 0 && n % group_size != 0)) return BAKRON_ERR_INVALID_ARG;
  for (int h = 0; h < H; ++h)
    if (!W[h] || !factors[h] || !codes[h] || !scales[h] || !zeros[h])
      return BAKRON_ERR_INVALID_ARG;
  const int S = streams < H ? streams : H;
  const size_t slice = slice_bytes(m, n);
  if (workspace_bytes < (size_t)S * slice) return BAKRON_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  // one enqueue at a time per process: the lanes and their events are shared
  std::lock_guard<std::mutex> lk(g_lanes_mu);
  Lanes* L = nullptr;
  int rc = lanes_for(S, &L);
  if (rc != BAKRON_OK) return rc;
  BK_CUDA_OK(cudaEventRecord(L->fork, s));
  // each lane clears its status word once; its solves keep the first error
  for (int l = 0; l < S; ++l) {
    BK_CUDA_OK(cudaStreamWaitEvent(L->stream[l], L->fork, 0));
    BK_CUDA_OK(cudaMemsetAsync(ws + (size_t)l * slice, 0, 256, L->stream[l]));
  }
  int launches = 0;
  bool done = false;
  if (S == H && H >= 2) {
    // one lane per problem: the leaves of all problems share one launch per
    // tile anti-diagonal on the caller's stream, the band products run per
    // problem on the lanes (unless the shape's schedule needs dataflow leaves
    // or persistent subtrees: then nothing was enqueued, and the lanes run
    // the problems one by one below)
    rc = solve_heads_impl(H, W, wdtype, m, n, ldw, factors, (1 << bits) - 1, group_size, codes,
                          scales, zeros, ws, slice, s, L->stream, L->fork, L->done);
    if (rc == BAKRON_ERR_INVALID_ARG) {
      rc = BAKRON_OK;
    } else {
      done = true;
      launches = launch_count();
    }
  }
  for (int h = 0; h < H && rc == BAKRON_OK && !done; ++h) {
    const int l = h % S;
    rc = solve_impl(W[h], wdtype, m, n, ldw, factors[h], (1 << bits) - 1, group_size, codes[h],
                    scales[h], zeros[h], nullptr, ws + (size_t)l * slice, L->stream[l], nullptr,
                    false, true);
    launches += launch_count();
  }
  // join every lane, also after a failed enqueue (what was enqueued stays ordered)
  for (int l = 0; l < S; ++l) {
    BK_CUDA_OK(cudaEventRecord(L->done[l], L->stream[l]));
    BK_CUDA_OK(cudaStreamWaitEvent(s, L->done[l], 0));
  }
  set_launch_count(launches);
  if (rc != BAKRON_OK || !sync) return rc;
  for (int l = 0; l < S; ++l) {
    const int st = bakron_read_status(ws + (size_t)l * slice, stream);
    if (st != BAKRON_OK && rc == BAKRON_OK) rc = st;
  }
  return rc;
}

int bakron_read_status_batched(void* workspace, int m, int n, int streams, void* stream) {
  if (!workspace || streams < 1 || streams > MAX_LANES || bakron_workspace_bytes(m, n) == 0)
    return BAKRON_ERR_INVALID_ARG;
  const size_t slice = slice_bytes(m, n);
  int rc = BAKRON_OK;
  for (int l = 0; l < streams; ++l) {
    const int st = bakron_read_status((char*)workspace + (size_t)l * slice, stream);
    if (st != BAKRON_OK && rc == BAKRON_OK) rc = st;
  }
  return rc;
}

}  // extern "C"
