// Isolated score + select + compaction without any device allocation.
//
// zsaa_score_select needs B*L floats of scratch for the row scores and takes
// them from the device's stream-ordered memory pool on every call.  Some
// callers cannot allocate device memory on their call path: serving loops that
// reserve their whole memory budget up front and treat any later allocation as
// a failure, latency-critical code that must not take the allocator's locks or
// its implicit synchronisation, and hosts whose framework owns every device
// allocation.  zsaa_score_select_noalloc serves them: its score scratch lives
// in the fixed array below, which the library holds on every GPU where its
// device code is loaded until the process exits.
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace {

// Largest B*L the allocation-free call accepts: 1,048,576 scores (4 MiB).
constexpr long long kNoAllocMaxScores = 1LL << 20;

static __device__ __align__(256) float g_noalloc_scores[kNoAllocMaxScores];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
float* g_scores_addr[kMaxDevices] = {};

}  // namespace

extern "C" zsaa_status zsaa_score_select_noalloc(const void* hidden, int B, int L, int d, int k,
                                                 int32_t* idx_out, void* gathered_out,
                                                 zsaa_stream stream) {
  char msg[160];
  if (static_cast<long long>(B) * static_cast<long long>(L) > kNoAllocMaxScores) {
    snprintf(msg, sizeof(msg),
             "zsaa_score_select_noalloc: B*L = %lld exceeds its fixed scratch of %lld scores",
             static_cast<long long>(B) * L, kNoAllocMaxScores);
    zsaa::set_last_error(msg);
    return ZSAA_ERR_INVALID_ARG;
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    snprintf(msg, sizeof(msg), "zsaa_score_select_noalloc: no usable current device (%s)",
             cudaGetErrorString(e));
    zsaa::set_last_error(msg);
    return ZSAA_ERR_CUDA;
  }
  float* scores = nullptr;
  {
    // First call on this device: look up the array's device address with the
    // device current.  In host code the array's name is only a stand-in.
    std::lock_guard<std::mutex> lk(g_setup_mu);
    if (g_scores_addr[dev] == nullptr) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_scores);
      if (e != cudaSuccess || p == nullptr) {
        snprintf(msg, sizeof(msg), "zsaa_score_select_noalloc: cudaGetSymbolAddress failed (%s)",
                 cudaGetErrorString(e));
        zsaa::set_last_error(msg);
        return ZSAA_ERR_CUDA;
      }
      g_scores_addr[dev] = static_cast<float*>(p);
    }
    scores = g_scores_addr[dev];
  }
  // Every score slot that the selection reads is rewritten first by the scoring
  // kernel, so nothing needs clearing between calls.
  return zsaa_score_select_ex(hidden, B, L, d, ZSAA_BF16, k, 0, nullptr, scores, idx_out,
                              gathered_out, stream);
}
