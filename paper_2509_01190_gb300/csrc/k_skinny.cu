// Weight-streaming GEMM for a few rows: out[M, N] = epi(A[M, K] W[N, K]^T), M <= 16.
//
// With at most 16 activation rows every weight is used at most 16 times, so the
// kernel is bound by reading W from HBM once.  Each CTA owns a 16-row band of W
// (grid-stride over bands); its 8 or 16 warps split K.  A warp streams its part of the
// band straight from global memory with 16-byte non-allocating loads, several
// 32-wide k chunks in flight, and multiplies on the tensor cores with
// mma.sync m16n8k16: the W band is the 16-row operand and the activation rows
// the 8-column one, so D[n, m] = sum_k W[n, k] A[m, k].
//
// Inside a 32-wide chunk the k order of the two MMAs is permuted so that each
// lane feeds them from one 16-byte load per W row and one per activation row:
// lane (g = lane/4, q = lane%4) loads k = 8q..8q+7, and MMA step s uses the pairs
// k = 8q+4s+{0,1} (fragment columns 2q, 2q+1) and 8q+4s+{2,3} (columns 2q+8,
// 2q+9) of both operands.  A dot product does not depend on the order of its
// terms, and both operands use the same permutation.
//
// The warps' partial sums are added in warp order in shared memory (a fixed
// order: results are deterministic), then the epilogue (bf16 store, residual
// add, SwiGLU, float32 store) writes the band.  Weights are read before waiting
// on the previous kernel (programmatic dependent launch): they are never written
// by the kernel that precedes this one on the stream.
#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {


__device__ __forceinline__ uint4 ld_stream(const bf16* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

__device__ __forceinline__ float silu_sk(float g) { return g / (1.f + __expf(-g)); }

// Two MMA steps (s = 0, 1) of one 32-wide chunk: w0 = row g, w8 = row g + 8 of
// the band, x = activation row; d accumulates D[n, m] for this lane's fragment.
__device__ __forceinline__ void mma_chunk(float (&d)[4], const uint4& w0, const uint4& w8,
                                          const uint4& x) {
  const uint32_t a0[4] = {w0.x, w8.x, w0.y, w8.y};
  mma_bf16_16816(d, a0, x.x, x.y);
  const uint32_t a1[4] = {w0.z, w8.z, w0.w, w8.w};
  mma_bf16_16816(d, a1, x.z, x.w);
}

// MF: activation fragments of 8 rows (1: M <= 8, 2: M <= 16).  U: chunks in flight.
template <int EPI, int MF, int U, int NW>
__global__ void __launch_bounds__(NW * 32, NW == 16 ? 1 : 2)
    skinny_gemm_kernel(const bf16* __restrict__ A, int lda, TcWeights W, GemmParams p, int bands) {
  pdl_trigger();
  constexpr bool DUAL = EPI == kEpiSwiGLU;
  constexpr int PER_LANE = 4 * MF * (DUAL ? 2 : 1);
  __shared__ float red[NW][PER_LANE * 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, q = lane & 3;
  const int K = p.K, M = p.M;
  const int chunks = K / 32;
  const int c_begin = warp * chunks / NW, c_end = (warp + 1) * chunks / NW;
  bool waited = false;

  for (int band = blockIdx.x; band < bands; band += gridDim.x) {
    const int n0 = band * 16;
    const bf16* wb;
    const bf16* wu = nullptr;
    if (DUAL) {
      wb = static_cast<const bf16*>(W.w0) + static_cast<size_t>(n0) * K;
      wu = static_cast<const bf16*>(W.w1) + static_cast<size_t>(n0) * K;
    } else if (n0 >= W.n2) {
      wb = static_cast<const bf16*>(W.w2) + static_cast<size_t>(n0 - W.n2) * K;
    } else if (n0 >= W.n1) {
      wb = static_cast<const bf16*>(W.w1) + static_cast<size_t>(n0 - W.n1) * K;
    } else {
      wb = static_cast<const bf16*>(W.w0) + static_cast<size_t>(n0) * K;
    }
    const bf16* wr0 = wb + static_cast<size_t>(g) * K + 8 * q;
    const bf16* wr8 = wr0 + static_cast<size_t>(8) * K;
    const bf16* ur0 = DUAL ? wu + static_cast<size_t>(g) * K + 8 * q : nullptr;
    const bf16* ur8 = DUAL ? ur0 + static_cast<size_t>(8) * K : nullptr;

    float acc[MF][4], accu[MF][4];
#pragma unroll
    for (int f = 0; f < MF; ++f)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[f][e] = accu[f][e] = 0.f;

    for (int c = c_begin; c < c_end; c += U) {
      uint4 w0[U], w8[U], u0[U], u8[U], x[U][MF];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (c + u < c_end) {
          const size_t k = static_cast<size_t>(c + u) * 32;
          w0[u] = ld_stream(wr0 + k);
          w8[u] = ld_stream(wr8 + k);
          if (DUAL) {
            u0[u] = ld_stream(ur0 + k);
            u8[u] = ld_stream(ur8 + k);
          }
        }
      }
      if (!waited) {  // activations come from the previous kernel
        pdl_wait();
        waited = true;
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (c + u < c_end) {
#pragma unroll
          for (int f = 0; f < MF; ++f) {
            const int m = 8 * f + g;
            x[u][f] = m < M ? *reinterpret_cast<const uint4*>(A + static_cast<size_t>(m) * lda +
                                                               (c + u) * 32 + 8 * q)
                            : make_uint4(0u, 0u, 0u, 0u);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (c + u < c_end) {
#pragma unroll
          for (int f = 0; f < MF; ++f) {
            mma_chunk(acc[f], w0[u], w8[u], x[u][f]);
            if (DUAL) mma_chunk(accu[f], u0[u], u8[u], x[u][f]);
          }
        }
      }
    }
    if (!waited) {  // a warp without chunks still orders its writes after the previous kernel
      pdl_wait();
      waited = true;
    }
    // partial sums of this warp -> shared memory; element e = lane * PER_LANE + j
#pragma unroll
    for (int f = 0; f < MF; ++f)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        red[warp][lane * PER_LANE + 4 * f + e] = acc[f][e];
        if (DUAL) red[warp][lane * PER_LANE + 4 * MF + 4 * f + e] = accu[f][e];
      }
    __syncthreads();
    for (int t = threadIdx.x; t < 32 * 4 * MF; t += NW * 32) {
      const int ln = t / (4 * MF), j = t % (4 * MF);
      const int f = j / 4, r = j % 4;
      const int n = n0 + (ln >> 2) + (r >= 2 ? 8 : 0);
      const int m = 8 * f + 2 * (ln & 3) + (r & 1);
      float v = 0.f, vu = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) {
        v += red[w][ln * PER_LANE + j];
        if (DUAL) vu += red[w][ln * PER_LANE + 4 * MF + j];
      }
      if (m >= M || n >= p.N) continue;
      const size_t o = static_cast<size_t>(m) * p.ldo + n;
      if (EPI == kEpiStoreF32) {
        static_cast<float*>(p.out)[o] = v;
      } else if (EPI == kEpiSwiGLU) {
        static_cast<bf16*>(p.out)[o] = __float2bfloat16_rn(silu_sk(v) * vu);
      } else if (EPI == kEpiResid) {
        const float r0 = __bfloat162float(static_cast<const bf16*>(p.resid)[o]);
        static_cast<bf16*>(p.out)[o] = __float2bfloat16_rn(r0 + v);
      } else {
        static_cast<bf16*>(p.out)[o] = __float2bfloat16_rn(v);
      }
    }
    __syncthreads();
  }
}

// SMs of the current device (kept per device).
int sm_count() {
  static int cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (cached[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    cached[dev] = n;
  }
  return cached[dev];
}

template <int EPI, int MF>
cudaError_t run_skinny(const bf16* A, int lda, const TcWeights& W, const GemmParams& p,
                       cudaStream_t s) {
  const int bands = p.N / 16;
  // chunks in flight per warp, as many as the registers allow: with 8 rows and
  // one weight matrix, a K = 2048 band's whole share (8 chunks) per round trip
  constexpr int U = EPI == kEpiSwiGLU ? (MF == 1 ? 4 : 2) : (MF == 1 ? 8 : 4);
  // deep K (>= 4096), one weight matrix and no more bands than SMs: 16 warps
  // split K (one CTA per SM and band), so each warp's share takes half the
  // round trips (1B down at 8 rows: 9.5 -> 7.3 us).  With more bands than
  // SMs the 8-warp form, two CTAs per SM, keeps every band on its own CTA.
  if (EPI != kEpiSwiGLU && MF == 1 && p.K >= 4096 && bands <= sm_count()) {
    ZSAA_LAUNCH(skinny_gemm_kernel<EPI, MF, U, 16>, dim3(bands), dim3(16 * 32), 0, s, A, lda, W, p, bands);
    return cudaSuccess;
  }
  const int cap = 2 * sm_count();
  const int grid = bands < cap ? bands : cap;
  ZSAA_LAUNCH(skinny_gemm_kernel<EPI, MF, U, 8>, dim3(grid), dim3(8 * 32), 0, s, A, lda, W, p, bands);
  return cudaSuccess;
}

template <int EPI>
cudaError_t run_skinny_m(const bf16* A, int lda, const TcWeights& W, const GemmParams& p,
                         cudaStream_t s) {
  return p.M <= 8 ? run_skinny<EPI, 1>(A, lda, W, p, s) : run_skinny<EPI, 2>(A, lda, W, p, s);
}

}  // namespace

bool skinny_supported(const void* A, int lda, const TcWeights& W, int epi, const GemmParams& p) {
  if (p.M < 1 || p.M > kSkinnyMaxM || epi == kEpiRope) return false;
  if (p.N % 16 != 0 || p.K % 32 != 0 || lda % 8 != 0) return false;
  if ((reinterpret_cast<uintptr_t>(A) & 15) != 0) return false;
  const void* ws[3] = {W.w0, W.w1, W.w2};
  for (const void* w : ws)
    if ((reinterpret_cast<uintptr_t>(w) & 15) != 0) return false;
  if (epi != kEpiSwiGLU && ((W.n1 % 16) != 0 || (W.n2 % 16) != 0)) return false;
  return true;
}

cudaError_t launch_gemm_skinny(const void* A, int lda, const TcWeights& W, int epi,
                               const GemmParams& p, cudaStream_t s) {
  if (p.launches) *p.launches += 1;
  const bf16* a = static_cast<const bf16*>(A);
  switch (epi) {
    case kEpiStore: return run_skinny_m<kEpiStore>(a, lda, W, p, s);
    case kEpiResid: return run_skinny_m<kEpiResid>(a, lda, W, p, s);
    case kEpiSwiGLU: return run_skinny_m<kEpiSwiGLU>(a, lda, W, p, s);
    case kEpiStoreF32: return run_skinny_m<kEpiStoreF32>(a, lda, W, p, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zsaa
