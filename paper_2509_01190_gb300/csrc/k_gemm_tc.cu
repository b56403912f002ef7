// bf16 GEMM on the sm_103a tensor cores: out = epi(A[M,K] W[N,K]^T), fp32
// accumulation in tensor memory.
//
// One CTA computes a 128 x BN tile with warp-specialised roles:
//   warp 0      TMA producer: 128B-swizzled A and W tiles (64 deep in K) into a
//               STAGES-deep shared-memory ring, completion on "full" mbarriers;
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16)
//               into a TMEM accumulator and frees each stage with
//               tcgen05.commit on its "empty" mbarrier;
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (each thread one row),
//               fused epilogue, 16-byte stores.
// Epilogues: bf16 store; residual add (h += acc, in place); SwiGLU (the tile's
// first BN/2 accumulator columns are gate rows of W, the last BN/2 up rows of
// W2; out = silu(gate) * up); float32 store (logits); RoPE of the query/key
// heads at each row's original position, then bf16 store.
// Every mbarrier wait is bounded (2 s); on expiry the kernel sets the status
// word, skips the remaining work and still frees its TMEM.
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr int BM = 128, BK = 64;
constexpr int kThreads = 192;

template <int BN>
struct TcCfg {
  static constexpr int STAGES = BN >= 256 ? 4 : (BN >= 128 ? 6 : 8);
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = BN;
  static constexpr size_t SMEM = static_cast<size_t>(STAGES) * STAGE_BYTES + 1024 + 256;
};

struct TcMaps {
  CUtensorMap a, b0, b1, b2;
};

__device__ __forceinline__ float silu_f(float g) { return g / (1.f + __expf(-g)); }

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ TcMaps maps, const int n1, const int n2,
                   const GemmParams p) {
  using C = TcCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* done = empty + C::STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int num_kb = p.K / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&maps.a);
    prefetch_tmap(&maps.b0);
    if (EPI == kEpiSwiGLU || n1 < p.N) prefetch_tmap(&maps.b1);
    if (n2 < p.N) prefetch_tmap(&maps.b2);
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      const CUtensorMap* mb = &maps.b0;
      int nb = n0;
      if (EPI != kEpiSwiGLU) {
        if (n0 >= n2) {
          mb = &maps.b2;
          nb = n0 - n2;
        } else if (n0 >= n1) {
          mb = &maps.b1;
          nb = n0 - n1;
        }
      }
      int issued = 0;
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % C::STAGES;
        const uint32_t ph = (kb / C::STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, p.status)) break;
        mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
        tma_load_2d(sA + s * C::A_BYTES, &maps.a, kb * BK, m0, &full[s]);
        if (EPI == kEpiSwiGLU) {
          tma_load_2d(sB + s * C::B_BYTES, &maps.b0, kb * BK, n0 / 2, &full[s]);
          tma_load_2d(sB + s * C::B_BYTES + (BN / 2) * 128, &maps.b1, kb * BK, n0 / 2, &full[s]);
        } else {
          tma_load_2d(sB + s * C::B_BYTES, mb, kb * BK, nb, &full[s]);
        }
        issued = kb + 1;
      }
      // Do not leave while copies into this CTA's shared memory may be in flight.
      for (int kb = issued - 1; kb >= 0 && kb >= issued - C::STAGES; --kb)
        mbar_wait(&full[kb % C::STAGES], (kb / C::STAGES) & 1, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % C::STAGES;
        const uint32_t ph = (kb / C::STAGES) & 1;
        if (!mbar_wait(&full[s], ph, p.status)) break;
        tc_fence_after();
        const uint32_t a_base = smem_u32(sA + s * C::A_BYTES);
        const uint32_t b_base = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          tc_mma_bf16(tmem, sdesc_sw128(a_base + k * 32), sdesc_sw128(b_base + k * 32), idesc,
                      (kb | k) != 0 ? 1u : 0u);
        tc_commit(&empty[s]);
      }
      tc_commit(done);
    }
    __syncwarp();
  } else {
    // Epilogue: warp w reads TMEM lanes 32*(w%4) .. +32, i.e. tile rows.
    const int quad = warp & 3;
    const int row = m0 + quad * 32 + lane;
    const bool row_ok = row < p.M;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const bool ok = __all_sync(0xffffffffu, mbar_wait(done, 0, p.status));
    tc_fence_after();
    if (ok) {
      if (EPI == kEpiSwiGLU) {
        bf16* out = static_cast<bf16*>(p.out);
        const int oc0 = n0 / 2;
#pragma unroll 1
        for (int c = 0; c < BN / 2; c += 16) {
          uint32_t g[16], u[16];
          __syncwarp();
          tmem_ld16(tbase + c, g);
          tmem_ld16(tbase + BN / 2 + c, u);
          tmem_ld_wait();
          if (row_ok && oc0 + c < p.N) {
            uint32_t o[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float g0 = __uint_as_float(g[2 * e]), g1 = __uint_as_float(g[2 * e + 1]);
              const float u0 = __uint_as_float(u[2 * e]), u1 = __uint_as_float(u[2 * e + 1]);
              o[e] = pack_bf16x2(silu_f(g0) * u0, silu_f(g1) * u1);
            }
            uint4* dst = reinterpret_cast<uint4*>(out + static_cast<size_t>(row) * p.ldo + oc0 + c);
            dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
            dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
          }
        }
      } else if (EPI == kEpiStoreF32) {
        float* out = static_cast<float*>(p.out);
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          uint32_t r[16];
          __syncwarp();
          tmem_ld16(tbase + c, r);
          tmem_ld_wait();
          if (row_ok && n0 + c < p.N) {
            uint4* dst = reinterpret_cast<uint4*>(out + static_cast<size_t>(row) * p.ldo + n0 + c);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              dst[q] = make_uint4(r[4 * q], r[4 * q + 1], r[4 * q + 2], r[4 * q + 3]);
          }
        }
      } else if (EPI == kEpiRope) {
        bf16* out = static_cast<bf16*>(p.out);
        const int hd = p.hd, half = hd / 2;
        const int ps = row_ok ? p.pos[row] : 0;
#pragma unroll 1
        for (int hs = 0; hs < BN; hs += hd) {
          const bool rot = n0 + hs < p.rope_cols;
#pragma unroll 1
          for (int c = 0; c < half; c += 16) {
            uint32_t x1[16], x2[16];
            __syncwarp();
            tmem_ld16(tbase + hs + c, x1);
            tmem_ld16(tbase + hs + half + c, x2);
            tmem_ld_wait();
            if (row_ok && n0 + hs < p.N) {
            float y1[16], y2[16];
            if (rot) {
              const float4* cp = reinterpret_cast<const float4*>(p.cos_t + static_cast<size_t>(ps) * half + c);
              const float4* sp = reinterpret_cast<const float4*>(p.sin_t + static_cast<size_t>(ps) * half + c);
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float4 cs = __ldg(cp + q), sn = __ldg(sp + q);
                const float cv[4] = {cs.x, cs.y, cs.z, cs.w}, sv[4] = {sn.x, sn.y, sn.z, sn.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float a = __uint_as_float(x1[4 * q + e]), b = __uint_as_float(x2[4 * q + e]);
                  y1[4 * q + e] = a * cv[e] - b * sv[e];
                  y2[4 * q + e] = b * cv[e] + a * sv[e];
                }
              }
            } else {
#pragma unroll
              for (int e = 0; e < 16; ++e) {
                y1[e] = __uint_as_float(x1[e]);
                y2[e] = __uint_as_float(x2[e]);
              }
            }
            uint32_t o1[8], o2[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              o1[e] = pack_bf16x2(y1[2 * e], y1[2 * e + 1]);
              o2[e] = pack_bf16x2(y2[2 * e], y2[2 * e + 1]);
            }
            bf16* rowp = out + static_cast<size_t>(row) * p.ldo + n0 + hs;
            uint4* d1 = reinterpret_cast<uint4*>(rowp + c);
            uint4* d2 = reinterpret_cast<uint4*>(rowp + half + c);
            d1[0] = make_uint4(o1[0], o1[1], o1[2], o1[3]);
            d1[1] = make_uint4(o1[4], o1[5], o1[6], o1[7]);
            d2[0] = make_uint4(o2[0], o2[1], o2[2], o2[3]);
            d2[1] = make_uint4(o2[4], o2[5], o2[6], o2[7]);
            }
          }
        }
      } else {  // kEpiStore / kEpiResid, bf16 out
        bf16* out = static_cast<bf16*>(p.out);
        const bf16* res = static_cast<const bf16*>(p.resid);
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          uint32_t r[16];
          __syncwarp();
          tmem_ld16(tbase + c, r);
          tmem_ld_wait();
          if (row_ok && n0 + c < p.N) {
            const size_t off = static_cast<size_t>(row) * p.ldo + n0 + c;
            float v[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) v[e] = __uint_as_float(r[e]);
            if (EPI == kEpiResid) {
              const uint4* rp = reinterpret_cast<const uint4*>(res + off);
              const uint4 r0 = rp[0], r1 = rp[1];
              const uint32_t rr[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
#pragma unroll
              for (int e = 0; e < 8; ++e) {
                v[2 * e] += bf16lo(rr[e]);
                v[2 * e + 1] += bf16hi(rr[e]);
              }
            }
            uint32_t o[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) o[e] = pack_bf16x2(v[2 * e], v[2 * e + 1]);
            uint4* dst = reinterpret_cast<uint4*>(out + off);
            dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
            dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

bool encode_2d(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint32_t box_rows) {
  EncodeTiledFn enc = get_encode_tiled();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                   box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int EPI>
cudaError_t run_tc(const TcMaps& maps, int n1, int n2, const GemmParams& p, int grid_n,
                   cudaStream_t s) {
  using C = TcCfg<BN>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(C::SMEM));
  });
  if (attr_err != cudaSuccess) return attr_err;
  dim3 grid(grid_n, (p.M + BM - 1) / BM);
  gemm_tc_kernel<BN, EPI><<<grid, kThreads, C::SMEM, s>>>(maps, n1, n2, p);
  return cudaGetLastError();
}

template <int BN>
cudaError_t dispatch_epi(int epi, const TcMaps& maps, int n1, int n2, const GemmParams& p,
                         int grid_n, cudaStream_t s) {
  switch (epi) {
    case kEpiStore: return run_tc<BN, kEpiStore>(maps, n1, n2, p, grid_n, s);
    case kEpiResid: return run_tc<BN, kEpiResid>(maps, n1, n2, p, grid_n, s);
    case kEpiSwiGLU: return run_tc<BN, kEpiSwiGLU>(maps, n1, n2, p, grid_n, s);
    case kEpiStoreF32: return run_tc<BN, kEpiStoreF32>(maps, n1, n2, p, grid_n, s);
    case kEpiRope: return run_tc<BN, kEpiRope>(maps, n1, n2, p, grid_n, s);
    default: return cudaErrorInvalidValue;
  }
}

bool bn_ok(int BN, int epi, const TcWeights& W, const GemmParams& p) {
  if (epi == kEpiSwiGLU) return true;
  if (W.n1 % BN != 0 && W.n1 < p.N) return false;
  if (W.n2 % BN != 0 && W.n2 < p.N) return false;
  if (epi == kEpiRope && (BN % p.hd != 0 || p.rope_cols % p.hd != 0)) return false;
  return true;
}

}  // namespace

cudaError_t launch_gemm_tc(const void* A, int lda, const TcWeights& W, int epi,
                           const GemmParams& p, cudaStream_t s) {
  if (p.K % BK != 0 || p.N % 16 != 0 || lda % 8 != 0) return cudaErrorInvalidValue;
  const int virtual_n = epi == kEpiSwiGLU ? 2 * p.N : p.N;
  const int m_tiles = (p.M + BM - 1) / BM;
  // Largest tile width that still gives about one wave of CTAs.
  int BN = 64;
  for (int cand : {256, 128}) {
    if (!bn_ok(cand, epi, W, p)) continue;
    const long tiles = static_cast<long>(m_tiles) * ((virtual_n + cand - 1) / cand);
    if (tiles >= 148) {
      BN = cand;
      break;
    }
  }
  if (!bn_ok(BN, epi, W, p)) BN = 128;
  if (!bn_ok(BN, epi, W, p)) return cudaErrorInvalidValue;

  TcMaps maps;
  memset(&maps, 0, sizeof(maps));
  const uint32_t brows = epi == kEpiSwiGLU ? BN / 2 : BN;
  if (!encode_2d(&maps.a, A, static_cast<uint64_t>(p.K), static_cast<uint64_t>(p.M), BM))
    return cudaErrorInvalidValue;
  if (lda != p.K) {
    // A is a column slice of a wider matrix: describe it with its own row stride.
    EncodeTiledFn enc = get_encode_tiled();
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(p.K), static_cast<cuuint64_t>(p.M)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(lda) * 2};
    cuuint32_t box[2] = {BK, BM};
    cuuint32_t es[2] = {1, 1};
    if (enc(&maps.a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(A), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  int n1 = W.n1, n2 = W.n2;
  if (epi == kEpiSwiGLU) {
    if (!encode_2d(&maps.b0, W.w0, p.K, p.N, brows)) return cudaErrorInvalidValue;
    if (!encode_2d(&maps.b1, W.w1, p.K, p.N, brows)) return cudaErrorInvalidValue;
    n1 = n2 = virtual_n;
  } else {
    const int r0 = n1 < p.N ? n1 : p.N;
    if (!encode_2d(&maps.b0, W.w0, p.K, r0, brows)) return cudaErrorInvalidValue;
    if (n1 < p.N) {
      const int r1 = (n2 < p.N ? n2 : p.N) - n1;
      if (!encode_2d(&maps.b1, W.w1, p.K, r1, brows)) return cudaErrorInvalidValue;
    }
    if (n2 < p.N) {
      if (!encode_2d(&maps.b2, W.w2, p.K, p.N - n2, brows)) return cudaErrorInvalidValue;
    }
  }
  const int grid_n = (virtual_n + BN - 1) / BN;
  switch (BN) {
    case 256: return dispatch_epi<256>(epi, maps, n1, n2, p, grid_n, s);
    case 128: return dispatch_epi<128>(epi, maps, n1, n2, p, grid_n, s);
    default: return dispatch_epi<64>(epi, maps, n1, n2, p, grid_n, s);
  }
}

}  // namespace zsaa
