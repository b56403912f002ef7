// bf16 GEMM on the sm_103a tensor cores: out = epi(A[M,K] W[N,K]^T), fp32
// accumulation in tensor memory.
//
// Persistent kernel: one CTA per SM walks a static list of 128 x BN tiles
// (tiles sharing a weight tile are adjacent, so weights stream from HBM once
// and are re-read from L2).  Warp-specialised roles:
//   warp 0      TMA producer: 128B-swizzled A and W tiles (64 deep in K) into a
//               STAGES-deep shared-memory ring ("full" mbarriers, expect-tx);
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16)
//               into one of two TMEM accumulators and frees each stage with
//               tcgen05.commit on its "empty" mbarrier;
//   warps 2..5  epilogue: tcgen05.ld of the finished accumulator (one row per
//               thread), fused epilogue, 16-byte stores; then they hand the
//               accumulator back, so the next tile's MMAs overlap this epilogue.
// Small problems split K: each split writes an fp32 partial tile to a
// workspace and splitk_finish_kernel sums the splits in a fixed order and
// applies the epilogue (deterministic, no atomics).
// Epilogues: bf16 store; residual add (h += acc, in place); SwiGLU (the tile's
// first BN/2 accumulator columns are gate rows of W, the last BN/2 up rows of
// W2; out = silu(gate) * up); float32 store (logits); RoPE of the query/key
// heads at each row's original position, then bf16 store.
// Every mbarrier wait is bounded (2 s); on expiry the kernel sets the status
// word, the other roles stop waiting, in-flight copies are drained (bounded)
// and TMEM is freed before the CTA exits.
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
  static constexpr int TMEM_COLS = 2 * BN;  // two accumulators
  static constexpr size_t SMEM = static_cast<size_t>(STAGES) * STAGE_BYTES + 1024 + 256;
};

struct TcMaps {
  CUtensorMap a, b0, b1, b2;
};

// Static tile list: tile t -> (m tile, n tile, K split), m fastest.
struct TileSched {
  int m_tiles, n_tiles, splits, kb_per_split, num_kb, total;
  float* ws;  // splits > 1: partial tiles [splits][M][VN] float32
  int vn;     // columns of the (virtual) product: N, or 2N for SwiGLU
};

__device__ __forceinline__ float silu_f(float g) { return g / (1.f + __expf(-g)); }

__device__ __forceinline__ void store_bf16x16(bf16* dst, const float (&v)[16]) {
  uint32_t o[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) o[e] = pack_bf16x2(v[2 * e], v[2 * e + 1]);
  uint4* d = reinterpret_cast<uint4*>(dst);
  d[0] = make_uint4(o[0], o[1], o[2], o[3]);
  d[1] = make_uint4(o[4], o[5], o[6], o[7]);
}

// Epilogue of one finished accumulator tile for this thread's row.
template <int BN, int EPI>
__device__ __forceinline__ void tile_epilogue(uint32_t tbase, int row, bool row_ok, int n0,
                                              const GemmParams& p, const TileSched& ts, int ks) {
  if (ts.splits > 1) {  // fp32 partial of this split, virtual column layout
    float* ws = ts.ws + (static_cast<size_t>(ks) * p.M + row) * ts.vn + n0;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      uint32_t r[32];
      __syncwarp();
      tmem_ld16(tbase + c, *reinterpret_cast<uint32_t(*)[16]>(r));
      tmem_ld16(tbase + c + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
      tmem_ld_wait();
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (row_ok && n0 + c + 16 * h < ts.vn) {
          uint4* dst = reinterpret_cast<uint4*>(ws + c + 16 * h);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            dst[q] = make_uint4(r[16 * h + 4 * q], r[16 * h + 4 * q + 1], r[16 * h + 4 * q + 2], r[16 * h + 4 * q + 3]);
        }
      }
    }
    return;
  }
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
        float v[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = silu_f(__uint_as_float(g[e])) * __uint_as_float(u[e]);
        store_bf16x16(out + static_cast<size_t>(row) * p.ldo + oc0 + c, v);
      }
    }
  } else if (EPI == kEpiStoreF32) {
    float* out = static_cast<float*>(p.out);
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      uint32_t r[32];
      __syncwarp();
      tmem_ld16(tbase + c, *reinterpret_cast<uint32_t(*)[16]>(r));
      tmem_ld16(tbase + c + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
      tmem_ld_wait();
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (row_ok && n0 + c + 16 * h < p.N) {
          uint4* dst = reinterpret_cast<uint4*>(out + static_cast<size_t>(row) * p.ldo + n0 + c + 16 * h);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            dst[q] = make_uint4(r[16 * h + 4 * q], r[16 * h + 4 * q + 1], r[16 * h + 4 * q + 2], r[16 * h + 4 * q + 3]);
        }
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
        float4 cs4[4], sn4[4];
        if (rot && row_ok) {  // table loads first: their latency overlaps the TMEM load
          const float4* cp = reinterpret_cast<const float4*>(p.cos_t + static_cast<size_t>(ps) * half + c);
          const float4* sp = reinterpret_cast<const float4*>(p.sin_t + static_cast<size_t>(ps) * half + c);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            cs4[q] = __ldg(cp + q);
            sn4[q] = __ldg(sp + q);
          }
        }
        __syncwarp();
        tmem_ld16(tbase + hs + c, x1);
        tmem_ld16(tbase + hs + half + c, x2);
        tmem_ld_wait();
        if (row_ok && n0 + hs < p.N) {
          float y1[16], y2[16];
          if (rot) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float4 cs = cs4[q], sn = sn4[q];
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
          bf16* rowp = out + static_cast<size_t>(row) * p.ldo + n0 + hs;
          store_bf16x16(rowp + c, y1);
          store_bf16x16(rowp + half + c, y2);
        }
      }
    }
  } else {  // kEpiStore / kEpiResid, bf16 out
    bf16* out = static_cast<bf16*>(p.out);
    const bf16* res = static_cast<const bf16*>(p.resid);
    const size_t rowoff = static_cast<size_t>(row) * p.ldo + n0;
    uint4 rc[4], rn[4];
    auto load_res = [&](int c, uint4 (&r)[4]) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (EPI == kEpiResid && row_ok && n0 + c + 16 * h < p.N) {
          const uint4* rp = reinterpret_cast<const uint4*>(res + rowoff + c + 16 * h);
          r[2 * h] = rp[0];
          r[2 * h + 1] = rp[1];
        } else {
          r[2 * h] = r[2 * h + 1] = make_uint4(0u, 0u, 0u, 0u);
        }
      }
    };
    load_res(0, rc);
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      if (c + 32 < BN) load_res(c + 32, rn);  // in flight while this chunk drains TMEM
      uint32_t r[32];
      __syncwarp();
      tmem_ld16(tbase + c, *reinterpret_cast<uint32_t(*)[16]>(r));
      tmem_ld16(tbase + c + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
      tmem_ld_wait();
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (row_ok && n0 + c + 16 * h < p.N) {
          float v[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] = __uint_as_float(r[16 * h + e]);
          if (EPI == kEpiResid) {
            const uint32_t rr[8] = {rc[2 * h].x, rc[2 * h].y, rc[2 * h].z, rc[2 * h].w,
                                    rc[2 * h + 1].x, rc[2 * h + 1].y, rc[2 * h + 1].z, rc[2 * h + 1].w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              v[2 * e] += bf16lo(rr[e]);
              v[2 * e + 1] += bf16hi(rr[e]);
            }
          }
          store_bf16x16(out + rowoff + c + 16 * h, v);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) rc[q] = rn[q];
    }
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ TcMaps maps, const int n1, const int n2,
                   const GemmParams p, const TileSched ts) {
  using C = TcCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* acc_full = empty + C::STAGES;  // [2]
  uint64_t* acc_empty = acc_full + 2;      // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);  // one arrival per epilogue warp
    }
    *abort_flag = 0;
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
      uint32_t it = 0, issued_last = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < ts.total && ok; t += gridDim.x) {
        const int mt = t % ts.m_tiles, r = t / ts.m_tiles;
        const int nt = r % ts.n_tiles, ks = r / ts.n_tiles;
        const int m0 = mt * BM, n0 = nt * BN;
        const int kb0 = ks * ts.kb_per_split;
        const int kb1 = min(ts.num_kb, kb0 + ts.kb_per_split);
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
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % C::STAGES;
          const uint32_t ph = (it / C::STAGES) & 1;
          if (!mbar_wait_ab(&empty[s], ph ^ 1, p.status, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
          tma_load_2d(sA + s * C::A_BYTES, &maps.a, kb * BK, m0, &full[s]);
          if (EPI == kEpiSwiGLU) {
            tma_load_2d(sB + s * C::B_BYTES, &maps.b0, kb * BK, n0 / 2, &full[s]);
            tma_load_2d(sB + s * C::B_BYTES + (BN / 2) * 128, &maps.b1, kb * BK, n0 / 2, &full[s]);
          } else {
            tma_load_2d(sB + s * C::B_BYTES, mb, kb * BK, nb, &full[s]);
          }
          issued_last = it + 1;
        }
      }
      // Do not leave while copies into this CTA's shared memory may be in flight.
      if (!ok || *abort_flag) {
        for (uint32_t j = issued_last; j > 0 && j + C::STAGES > issued_last; --j) {
          const uint32_t q = j - 1;
          mbar_wait(&full[q % C::STAGES], (q / C::STAGES) & 1, nullptr);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      uint32_t it = 0;
      bool ok = true;
      int i = 0;
      for (int t = blockIdx.x; t < ts.total && ok; t += gridDim.x, ++i) {
        const int r = t / ts.m_tiles;
        const int ks = r / ts.n_tiles;
        const int kb0 = ks * ts.kb_per_split;
        const int kb1 = min(ts.num_kb, kb0 + ts.kb_per_split);
        const int ab = i & 1;
        const uint32_t use = static_cast<uint32_t>(i >> 1);
        if (!mbar_wait_ab(&acc_empty[ab], (use & 1) ^ 1, p.status, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(ab * BN);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % C::STAGES;
          const uint32_t ph = (it / C::STAGES) & 1;
          if (!mbar_wait_ab(&full[s], ph, p.status, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b_base = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma_bf16(d_tmem, sdesc_sw128(a_base + k * 32), sdesc_sw128(b_base + k * 32), idesc,
                        (kb > kb0 || k > 0) ? 1u : 0u);
          tc_commit(&empty[s]);
        }
        tc_commit(&acc_full[ab]);
      }
    }
    __syncwarp();
  } else {
    // Epilogue: warp w reads TMEM lanes 32*(w%4) .. +32, i.e. tile rows.
    const int quad = warp & 3;
    int i = 0;
    for (int t = blockIdx.x; t < ts.total; t += gridDim.x, ++i) {
      const int mt = t % ts.m_tiles, r = t / ts.m_tiles;
      const int nt = r % ts.n_tiles, ks = r / ts.n_tiles;
      const int row = mt * BM + quad * 32 + lane;
      const int ab = i & 1;
      const uint32_t use = static_cast<uint32_t>(i >> 1);
      const bool ok = __all_sync(0xffffffffu, mbar_wait_ab(&acc_full[ab], use & 1, p.status, abort_flag));
      if (!ok) break;
      tc_fence_after();
      const uint32_t tbase = tmem + static_cast<uint32_t>(ab * BN) + (static_cast<uint32_t>(quad * 32) << 16);
      tile_epilogue<BN, EPI>(tbase, row, row < p.M, nt * BN, p, ts, ks);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acc_empty[ab])) : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// Sum the K splits in order and apply the epilogue.  One thread per 8 output
// columns of one row (RoPE: per 8 rotation pairs of one head).
template <int EPI>
__global__ void splitk_finish_kernel(const float* __restrict__ ws, int splits, int BN,
                                     const GemmParams p, int vn) {
  const int row = blockIdx.y;
  const int ncols = EPI == kEpiRope ? p.rope_cols / 2 + (p.N - p.rope_cols) : p.N;
  const int chunk = blockIdx.x * blockDim.x + threadIdx.x;
  if (row >= p.M || chunk * 8 >= ncols) return;
  const size_t plane = static_cast<size_t>(p.M) * vn;
  const float* base = ws + static_cast<size_t>(row) * vn;
  auto sum8 = [&](int col, float (&v)[8]) {
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = 0.f;
    for (int s = 0; s < splits; ++s) {
      const float4* q = reinterpret_cast<const float4*>(base + s * plane + col);
      const float4 a = q[0], b = q[1];
      v[0] += a.x; v[1] += a.y; v[2] += a.z; v[3] += a.w;
      v[4] += b.x; v[5] += b.y; v[6] += b.z; v[7] += b.w;
    }
  };
  auto put_bf16 = [&](bf16* dst, const float (&v)[8]) {
    *reinterpret_cast<uint4*>(dst) = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                                pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
  };
  if (EPI == kEpiSwiGLU) {
    const int c = chunk * 8, half = BN / 2;
    const int vcol = (c / half) * BN + c % half;
    float g[8], u[8], v[8];
    sum8(vcol, g);
    sum8(vcol + half, u);
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = silu_f(g[e]) * u[e];
    put_bf16(static_cast<bf16*>(p.out) + static_cast<size_t>(row) * p.ldo + c, v);
  } else if (EPI == kEpiRope) {
    const int pairs = p.rope_cols / 2;
    const int half = p.hd / 2;
    bf16* out = static_cast<bf16*>(p.out) + static_cast<size_t>(row) * p.ldo;
    if (chunk * 8 < pairs) {
      const int pr = chunk * 8, head = pr / half, c = pr % half;
      const int col1 = head * p.hd + c, col2 = col1 + half;
      float x1[8], x2[8], y1[8], y2[8];
      sum8(col1, x1);
      sum8(col2, x2);
      const int ps = p.pos[row];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float cs = p.cos_t[static_cast<size_t>(ps) * half + c + e];
        const float sn = p.sin_t[static_cast<size_t>(ps) * half + c + e];
        y1[e] = x1[e] * cs - x2[e] * sn;
        y2[e] = x2[e] * cs + x1[e] * sn;
      }
      put_bf16(out + col1, y1);
      put_bf16(out + col2, y2);
    } else {
      const int col = p.rope_cols + (chunk * 8 - pairs);
      float v[8];
      sum8(col, v);
      put_bf16(out + col, v);
    }
  } else {
    const int c = chunk * 8;
    float v[8];
    sum8(c, v);
    const size_t off = static_cast<size_t>(row) * p.ldo + c;
    if (EPI == kEpiStoreF32) {
      float4* d = reinterpret_cast<float4*>(static_cast<float*>(p.out) + off);
      d[0] = make_float4(v[0], v[1], v[2], v[3]);
      d[1] = make_float4(v[4], v[5], v[6], v[7]);
    } else {
      if (EPI == kEpiResid) {
        const uint4 r = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(p.resid) + off);
        const uint32_t rr[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          v[2 * e] += bf16lo(rr[e]);
          v[2 * e + 1] += bf16hi(rr[e]);
        }
      }
      put_bf16(static_cast<bf16*>(p.out) + off, v);
    }
  }
}

bool encode_2d(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint64_t row_elems,
               uint32_t box_rows) {
  EncodeTiledFn enc = get_encode_tiled();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_elems * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                   box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int num_sms() {
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

template <int BN, int EPI>
cudaError_t run_tc(const TcMaps& maps, int n1, int n2, const GemmParams& p, const TileSched& ts,
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
  const int grid = ts.total < num_sms() ? ts.total : num_sms();
  gemm_tc_kernel<BN, EPI><<<grid, kThreads, C::SMEM, s>>>(maps, n1, n2, p, ts);
  cudaError_t e = cudaGetLastError();
  if (p.launches) *p.launches += 1;
  if (e != cudaSuccess || ts.splits == 1) return e;
  if (p.launches) *p.launches += 1;
  const int ncols = EPI == kEpiRope ? p.rope_cols / 2 + (p.N - p.rope_cols) : p.N;
  const int chunks = (ncols + 7) / 8;
  dim3 fgrid((chunks + 127) / 128, p.M);
  splitk_finish_kernel<EPI><<<fgrid, 128, 0, s>>>(ts.ws, ts.splits, BN, p, ts.vn);
  return cudaGetLastError();
}

template <int BN>
cudaError_t dispatch_epi(int epi, const TcMaps& maps, int n1, int n2, const GemmParams& p,
                         const TileSched& ts, cudaStream_t s) {
  switch (epi) {
    case kEpiStore: return run_tc<BN, kEpiStore>(maps, n1, n2, p, ts, s);
    case kEpiResid: return run_tc<BN, kEpiResid>(maps, n1, n2, p, ts, s);
    case kEpiSwiGLU: return run_tc<BN, kEpiSwiGLU>(maps, n1, n2, p, ts, s);
    case kEpiStoreF32: return run_tc<BN, kEpiStoreF32>(maps, n1, n2, p, ts, s);
    case kEpiRope: return run_tc<BN, kEpiRope>(maps, n1, n2, p, ts, s);
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
  const int sms = num_sms();
  const int vn = epi == kEpiSwiGLU ? 2 * p.N : p.N;
  const int m_tiles = (p.M + BM - 1) / BM;
  // Widest tile that still gives a full wave; otherwise the narrowest legal one.
  int BN = 0;
  for (int cand : {256, 128, 64}) {
    if (!bn_ok(cand, epi, W, p)) continue;
    BN = cand;
    if (static_cast<long>(m_tiles) * ((vn + cand - 1) / cand) >= sms) break;
  }
  if (BN == 0) return cudaErrorInvalidValue;
  TileSched ts{};
  ts.m_tiles = m_tiles;
  ts.n_tiles = (vn + BN - 1) / BN;
  ts.num_kb = p.K / BK;
  ts.vn = vn;
  ts.splits = 1;
  const long tiles = static_cast<long>(ts.m_tiles) * ts.n_tiles;
  // Split K while the tiles fill less than one wave and each split keeps >= 4 k-blocks.
  if (p.splitk_ws != nullptr) {
    while (tiles * ts.splits < sms && ts.num_kb / (2 * ts.splits) >= 4 &&
           static_cast<size_t>(2 * ts.splits) * p.M * vn <= p.splitk_ws_elems)
      ts.splits *= 2;
  }
  ts.kb_per_split = (ts.num_kb + ts.splits - 1) / ts.splits;
  ts.splits = (ts.num_kb + ts.kb_per_split - 1) / ts.kb_per_split;
  ts.total = static_cast<int>(tiles * ts.splits);
  ts.ws = p.splitk_ws;

  TcMaps maps;
  memset(&maps, 0, sizeof(maps));
  const uint32_t brows = epi == kEpiSwiGLU ? BN / 2 : BN;
  if (!encode_2d(&maps.a, A, static_cast<uint64_t>(p.K), static_cast<uint64_t>(p.M),
                 static_cast<uint64_t>(lda), BM))
    return cudaErrorInvalidValue;
  int n1 = W.n1, n2 = W.n2;
  if (epi == kEpiSwiGLU) {
    if (!encode_2d(&maps.b0, W.w0, p.K, p.N, p.K, brows)) return cudaErrorInvalidValue;
    if (!encode_2d(&maps.b1, W.w1, p.K, p.N, p.K, brows)) return cudaErrorInvalidValue;
    n1 = n2 = vn;
  } else {
    const int r0 = n1 < p.N ? n1 : p.N;
    if (!encode_2d(&maps.b0, W.w0, p.K, r0, p.K, brows)) return cudaErrorInvalidValue;
    if (n1 < p.N) {
      const int r1 = (n2 < p.N ? n2 : p.N) - n1;
      if (!encode_2d(&maps.b1, W.w1, p.K, r1, p.K, brows)) return cudaErrorInvalidValue;
    }
    if (n2 < p.N) {
      if (!encode_2d(&maps.b2, W.w2, p.K, p.N - n2, p.K, brows)) return cudaErrorInvalidValue;
    }
  }
  switch (BN) {
    case 256: return dispatch_epi<256>(epi, maps, n1, n2, p, ts, s);
    case 128: return dispatch_epi<128>(epi, maps, n1, n2, p, ts, s);
    default: return dispatch_epi<64>(epi, maps, n1, n2, p, ts, s);
  }
}

}  // namespace zsaa
