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

// The array's device address belongs to the context that loaded the module.
// After cudaDeviceReset (or any reset of the primary context) the module is
// loaded again in a new context, so the address is cached together with the
// id of the context it was looked up in, and looked up again when it changes.
struct ScratchAddr {
  unsigned long long ctx_id = 0;
  float* ptr = nullptr;
};
std::mutex g_setup_mu;
ScratchAddr g_scores_addr[kMaxDevices];

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// The id of the current context (0 if there is none or the driver lacks the call).
unsigned long long current_ctx_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(fn);
    fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(fn);
  });
  if (get_current == nullptr || get_id == nullptr) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

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
    // First call on this device (or in a new context of it): look up the
    // array's device address with the device current.  In host code the
    // array's name is only a stand-in.
    std::lock_guard<std::mutex> lk(g_setup_mu);
    ScratchAddr& slot = g_scores_addr[dev];
    const unsigned long long id = current_ctx_id();
    if (slot.ptr == nullptr || id == 0 || id != slot.ctx_id) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_scores);
      if (e != cudaSuccess || p == nullptr) {
        snprintf(msg, sizeof(msg), "zsaa_score_select_noalloc: cudaGetSymbolAddress failed (%s)",
                 cudaGetErrorString(e));
        zsaa::set_last_error(msg);
        return ZSAA_ERR_CUDA;
      }
      slot.ptr = static_cast<float*>(p);
      slot.ctx_id = current_ctx_id();  // the lookup made the context current if it was not
    }
    scores = slot.ptr;
  }
  // Every score slot that the selection reads is rewritten first by the scoring
  // kernel, so nothing needs clearing between calls.
  return zsaa_score_select_ex(hidden, B, L, d, ZSAA_BF16, k, 0, nullptr, scores, idx_out,
                              gathered_out, stream);
}
