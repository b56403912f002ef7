// fp32 CUDA-core GEMM for models stored in float32: out = epi(A[M,K] W[N,K]^T).
// True fp32 FMA (no TF32), 64x64 tiles, 4x4 outputs per thread.  Epilogues:
// store, residual add, SwiGLU (two weight matrices, gate and up).
#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr int TB = 64, TK = 16;

template <bool DUAL>
__global__ void __launch_bounds__(256)
    gemm_f32_kernel(const float* __restrict__ A, int lda, const float* __restrict__ W,
                    const float* __restrict__ W2, int M, int N, int K, int epi,
                    float* __restrict__ out, int ldo, const float* resid) {
  pdl_trigger();
  pdl_wait();
  __shared__ float As[TK][TB + 4];
  __shared__ float Ws[TK][TB + 4];
  __shared__ float W2s[DUAL ? TK : 1][TB + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * TB, n0 = blockIdx.x * TB;
  float acc[4][4] = {}, acc2[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int i = threadIdx.x; i < TB * TK; i += 256) {
      const int r = i / TK, c = i % TK;
      const bool kin = k0 + c < K;
      As[c][r] = (m0 + r < M && kin) ? A[static_cast<size_t>(m0 + r) * lda + k0 + c] : 0.f;
      Ws[c][r] = (n0 + r < N && kin) ? W[static_cast<size_t>(n0 + r) * K + k0 + c] : 0.f;
      if (DUAL) W2s[c][r] = (n0 + r < N && kin) ? W2[static_cast<size_t>(n0 + r) * K + k0 + c] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], w[4], w2[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        w[i] = Ws[kk][tx * 4 + i];
        if (DUAL) w2[i] = W2s[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
          if (DUAL) acc2[i][j] = fmaf(a[i], w2[j], acc2[i][j]);
        }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= N) continue;
      const size_t o = static_cast<size_t>(m) * ldo + n;
      float v = acc[i][j];
      if (DUAL) {
        const float g = v;
        v = g / (1.f + expf(-g)) * acc2[i][j];
      } else if (epi == kEpiResid) {
        v += resid[o];
      }
      out[o] = v;
    }
  }
}

}  // namespace

cudaError_t launch_gemm_f32(const float* A, int lda, const float* W, const float* W2, int epi,
                            const GemmParams& p, cudaStream_t s) {
  if (p.launches) *p.launches += 1;
  dim3 grid((p.N + TB - 1) / TB, (p.M + TB - 1) / TB);
  if (epi == kEpiSwiGLU)
    ZSAA_LAUNCH(gemm_f32_kernel<true>, dim3(grid), dim3(256), 0, s, A, lda, W, W2, p.M, p.N, p.K, epi,
                                               static_cast<float*>(p.out), p.ldo,
                                               static_cast<const float*>(p.resid));
  else
    ZSAA_LAUNCH(gemm_f32_kernel<false>, dim3(grid), dim3(256), 0, s, A, lda, W, nullptr, p.M, p.N, p.K, epi,
                                                static_cast<float*>(p.out), p.ldo,
                                                static_cast<const float*>(p.resid));
  return cudaGetLastError();
}

}  // namespace zsaa
