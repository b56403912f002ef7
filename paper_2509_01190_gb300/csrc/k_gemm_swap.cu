// bf16 GEMM for few rows on the sm_103a tensor cores, operands swapped:
// out[M, N] = epi(A[M, K] W[N, K]^T) computed as D[n, m] = W[n, :] . A[m, :].
//
// When the pruned prefill has kept only a few hundred rows, 128-row activation
// tiles leave the tile grid small (tens of CTAs), and every CTA streams its
// whole activation tile and weight band through one long serial K loop.  Here
// the weight band is the 128-row tcgen05 operand and the activation rows the
// MMA's N side (16..256 of them), so one MMA consumes a weight tile once for
// every row, and K is split over a thread-block cluster of S CTAs:
//   grid (S, bands, row blocks), cluster (S, 1, 1); CTA r of a cluster owns
//   k-blocks [r nkb / S, (r + 1) nkb / S) of one 128-row weight band
//   (SwiGLU: 64 gate rows of W and the same 64 up rows of W2) and one block
//   of at most 256 activation rows.
// Roles in a CTA of 512 threads:
//   warp 0      TMA producer: the 128-byte-swizzled weight tile [128 x 64] and
//               activation tile [Mp x 64] of each k-block into a ring of
//               shared-memory stages (weights are requested before waiting for
//               the previous kernel: no kernel writes them);
//   warp 1      MMA issuer: tcgen05.mma M=128, N=Mp, K=16 into one TMEM
//               accumulator [128 lanes x Mp columns];
//   warps 2..9  copy the finished partial accumulator into shared memory as
//               red[m][n] (fp32), reusing the drained stage ring;
//   all 16 warps then share the reduction and epilogue (one CTA fits an SM,
//               so the extra warps cost nothing and hide the latencies).
// A cluster barrier makes every CTA's partial visible; CTA r then adds the S
// partials of its share of the rows, in rank order over distributed shared
// memory (deterministic, no global workspace, no atomics), applies the
// epilogue -- bf16 store, residual add, SwiGLU, float32 store, RoPE with the
// value-head norms -- and writes full 256-byte row segments.  A second cluster
// barrier keeps every CTA's shared memory alive until the others have read it.
// Every mbarrier wait is bounded (2 s): on expiry the status word is set, the
// roles stop, in-flight copies are drained and every thread still reaches both
// cluster barriers, so no CTA of the cluster waits forever.
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>

#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr int SW_BK = 64;
constexpr int SW_BAND = 128;  // weight rows per CTA: the tcgen05 M
constexpr int SW_THREADS = 512;
constexpr int SW_WARPS = SW_THREADS / 32;
constexpr int SW_DRAIN_WARPS = 8;  // warps 2..9 copy the accumulator out of TMEM
constexpr int SW_W_BYTES = SW_BAND * SW_BK * 2;
constexpr int SW_MAX_CLUSTER = 8;
constexpr int SW_RING_BUDGET = 220 * 1024;  // bytes of stage ring per CTA
constexpr int SW_MAX_STAGES = 8;

struct SwMaps {
  CUtensorMap x, w0, w1, w2;
};

struct SwShape {
  int Mp;         // activation rows per row block (multiple of 16, <= 256): the MMA's N
  int stages;     // depth of the stage ring
  int ksub;       // k-blocks of 64 per stage
  int nkb;        // k-blocks of 64
  int n1, n2;     // weight row blocks (non-SwiGLU): w0 [0, n1), w1 [n1, n2), w2 [n2, N)
  uint32_t tmem_cols;
};

__device__ __forceinline__ float4 ld_dsmem_v4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}
__device__ __forceinline__ float2 ld_dsmem_v2(uint32_t addr) {
  float2 v;
  asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ float silu_sw(float g) { return g / (1.f + __expf(-g)); }

__device__ __forceinline__ float4 f4_add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 f4_shfl_xor(float4 v, int o) {
  v.x = __shfl_xor_sync(0xffffffffu, v.x, o);
  v.y = __shfl_xor_sync(0xffffffffu, v.y, o);
  v.z = __shfl_xor_sync(0xffffffffu, v.z, o);
  v.w = __shfl_xor_sync(0xffffffffu, v.w, o);
  return v;
}
__device__ __forceinline__ uint2 pack4_bf16(float4 v) {
  return make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
}
__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// Finish rows [m_lo, m_hi) of this block (a warp per row, RB rows of a warp in
// flight): add the cluster's partial sums in rank order, apply the epilogue,
// store.  LOCAL: the cluster is this CTA alone and red is read directly.
template <int EPI, int RB, bool LOCAL>
__device__ __forceinline__ void swap_epilogue(const GemmParams& p, const float* red,
                                              const uint32_t (&src)[SW_MAX_CLUSTER], int S, int band,
                                              int row0, int m_lo, int m_hi, int warp, int lane) {
  constexpr int STEP = RB * SW_WARPS;
  if (EPI == kEpiSwiGLU) {
    // lanes: output columns band*64 + 2*lane, +1 (gate in red columns 0..63, up in 64..127)
    bf16* out = static_cast<bf16*>(p.out);
    const int col = band * (SW_BAND / 2) + 2 * lane;
#pragma unroll 1
    for (int m = m_lo + warp; m < m_hi; m += STEP) {
      float2 g[RB], u[RB];
      if (LOCAL) {
#pragma unroll
        for (int r = 0; r < RB; ++r) {
          const int mr = min(m + r * SW_WARPS, m_hi - 1);
          g[r] = *reinterpret_cast<const float2*>(red + mr * SW_BAND + 2 * lane);
          u[r] = *reinterpret_cast<const float2*>(red + mr * SW_BAND + SW_BAND / 2 + 2 * lane);
        }
      } else {
        float2 tg[RB][SW_MAX_CLUSTER], tu[RB][SW_MAX_CLUSTER];
#pragma unroll
        for (int c = 0; c < SW_MAX_CLUSTER; ++c)
          if (c < S) {
#pragma unroll
            for (int r = 0; r < RB; ++r) {
              const uint32_t o = static_cast<uint32_t>(min(m + r * SW_WARPS, m_hi - 1) * SW_BAND + 2 * lane) * 4u;
              tg[r][c] = ld_dsmem_v2(src[c] + o);
              tu[r][c] = ld_dsmem_v2(src[c] + o + 4u * (SW_BAND / 2));
            }
          }
#pragma unroll
        for (int r = 0; r < RB; ++r) {
          g[r] = tg[r][0];
          u[r] = tu[r][0];
#pragma unroll
          for (int c = 1; c < SW_MAX_CLUSTER; ++c)
            if (c < S) {
              g[r] = make_float2(g[r].x + tg[r][c].x, g[r].y + tg[r][c].y);
              u[r] = make_float2(u[r].x + tu[r][c].x, u[r].y + tu[r][c].y);
            }
        }
      }
#pragma unroll
      for (int r = 0; r < RB; ++r) {
        const int mr = m + r * SW_WARPS;
        if (mr < m_hi && col < p.N)
          *reinterpret_cast<uint32_t*>(out + static_cast<size_t>(row0 + mr) * p.ldo + col) =
              pack_bf16x2(silu_sw(g[r].x) * u[r].x, silu_sw(g[r].y) * u[r].y);
      }
    }
    return;
  }
  const int n0 = band * SW_BAND;
  const int nl = 4 * lane;  // this lane's 4 columns of the band
  const int ncol = n0 + nl;
  // RoPE: the head of these columns, and the positions of this warp's first
  // 32 rows (lane t holds that of its row t)
  const int hd = EPI == kEpiRope ? p.hd : SW_BAND;
  const int half = hd / 2, j = nl % hd, hs = nl - j;
  const bool rot = EPI == kEpiRope && n0 + hs < p.rope_cols;
  const int jj = j < half ? j : j - half;
  int pos_lane = 0;
  if (EPI == kEpiRope) {
    const int mr = m_lo + warp + SW_WARPS * lane;
    if (mr < m_hi) pos_lane = p.pos[row0 + mr];
  }
  int t = 0;  // row counter of this warp: m = m_lo + warp + SW_WARPS * t
#pragma unroll 1
  for (int m = m_lo + warp; m < m_hi; m += STEP, t += RB) {
    // operands of the epilogue other than the accumulator
    uint2 rr[RB];
    float4 cs[RB], sn[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      rr[r] = make_uint2(0u, 0u);
      cs[r] = make_float4(1.f, 1.f, 1.f, 1.f);
      sn[r] = make_float4(0.f, 0.f, 0.f, 0.f);
      const int mr = m + r * SW_WARPS;
      const bool ok = mr < m_hi;
      if (EPI == kEpiResid && ok && ncol < p.N)
        rr[r] = *reinterpret_cast<const uint2*>(static_cast<const bf16*>(p.resid) +
                                                static_cast<size_t>(row0 + mr) * p.ldo + ncol);
      if (EPI == kEpiRope) {
        int ps = __shfl_sync(0xffffffffu, pos_lane, (t + r) & 31);
        if (t + r >= 32 && ok) ps = p.pos[row0 + mr];
        if (rot && ok) {
          cs[r] = __ldg(reinterpret_cast<const float4*>(p.cos_t + static_cast<size_t>(ps) * half + jj));
          sn[r] = __ldg(reinterpret_cast<const float4*>(p.sin_t + static_cast<size_t>(ps) * half + jj));
        }
      }
    }
    float4 v[RB];
    if (LOCAL) {
#pragma unroll
      for (int r = 0; r < RB; ++r)
        v[r] = *reinterpret_cast<const float4*>(red + min(m + r * SW_WARPS, m_hi - 1) * SW_BAND + nl);
    } else {
      float4 tv[RB][SW_MAX_CLUSTER];
#pragma unroll
      for (int c = 0; c < SW_MAX_CLUSTER; ++c)
        if (c < S) {
#pragma unroll
          for (int r = 0; r < RB; ++r)
            tv[r][c] = ld_dsmem_v4(src[c] + static_cast<uint32_t>(min(m + r * SW_WARPS, m_hi - 1) * SW_BAND + nl) * 4u);
        }
#pragma unroll
      for (int r = 0; r < RB; ++r) {
        v[r] = tv[r][0];
#pragma unroll
        for (int c = 1; c < SW_MAX_CLUSTER; ++c)
          if (c < S) v[r] = f4_add(v[r], tv[r][c]);
      }
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int mr = m + r * SW_WARPS;
      if (mr >= m_hi) break;  // warp-uniform
      const int row = row0 + mr;
      const size_t o = static_cast<size_t>(row) * p.ldo + ncol;
      if (EPI == kEpiStoreF32) {
        if (ncol < p.N) *reinterpret_cast<float4*>(static_cast<float*>(p.out) + o) = v[r];
      } else if (EPI == kEpiRope) {
        // the rotation pairs column j of a head with column j + hd/2: hd/8 lanes apart
        const float4 x = v[r], w = f4_shfl_xor(x, hd / 8), c4 = cs[r], s4 = sn[r];
        float4 y = x;
        if (rot) {
          if (j < half) {
            y = make_float4(x.x * c4.x - w.x * s4.x, x.y * c4.y - w.y * s4.y, x.z * c4.z - w.z * s4.z,
                            x.w * c4.w - w.w * s4.w);
          } else {
            y = make_float4(x.x * c4.x + w.x * s4.x, x.y * c4.y + w.y * s4.y, x.z * c4.z + w.z * s4.z,
                            x.w * c4.w + w.w * s4.w);
          }
        }
        if (ncol < p.N) *reinterpret_cast<uint2*>(static_cast<bf16*>(p.out) + o) = pack4_bf16(y);
        if (p.vnorm_out != nullptr) {
          // ||v|| of a value head over its stored (bf16) values: hd/4 lanes per head
          float ss = 0.f;
          if (!rot) {
            const float a = bf16_round(y.x), b = bf16_round(y.y), c = bf16_round(y.z), d = bf16_round(y.w);
            ss = a * a + b * b + c * c + d * d;
          }
          for (int w2 = 1; w2 < hd / 4; w2 <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, w2);
          if (!rot && j == 0 && n0 + hs < p.N) {
            const int groups = (p.N - p.rope_cols) / hd;
            p.vnorm_out[static_cast<size_t>(row) * groups + (n0 + hs - p.rope_cols) / hd] = sqrtf(ss);
          }
        }
      } else {
        float4 x = v[r];
        if (EPI == kEpiResid) {
          x.x += bf16lo(rr[r].x);
          x.y += bf16hi(rr[r].x);
          x.z += bf16lo(rr[r].y);
          x.w += bf16hi(rr[r].y);
        }
        if (ncol < p.N) *reinterpret_cast<uint2*>(static_cast<bf16*>(p.out) + o) = pack4_bf16(x);
      }
    }
  }
}

template <int EPI>
__global__ void __launch_bounds__(SW_THREADS, 1)
    gemm_swap_kernel(const __grid_constant__ SwMaps maps, const SwShape sh, const GemmParams p) {
  constexpr bool DUAL = EPI == kEpiSwiGLU;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int X_BYTES = sh.Mp * SW_BK * 2;  // one activation sub-tile [Mp x 64]
  const int WSUB = SW_W_BYTES;  // weight bytes of one k-block
  const int STAGES = sh.stages, KSUB = sh.ksub;
  uint8_t* sW = smem;                                     // [STAGES][KSUB] weight sub-tiles
  uint8_t* sX = smem + STAGES * KSUB * WSUB;              // [STAGES][KSUB] activation sub-tiles
  uint64_t* full = reinterpret_cast<uint64_t*>(sX + STAGES * KSUB * X_BYTES);
  uint64_t* empty = full + SW_MAX_STAGES;
  uint64_t* acc_full = empty + SW_MAX_STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* red = reinterpret_cast<float*>(smem);  // [Mp][128] fp32, over the drained ring

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = static_cast<int>(cluster_size()), rank = static_cast<int>(cluster_rank());
  const int band = blockIdx.y;
  const int row0 = blockIdx.z * sh.Mp;                       // first activation row of this block
  const int rows = min(sh.Mp, p.M - row0);                   // valid rows of this block
  const int kb0 = rank * sh.nkb / S, kb1 = (rank + 1) * sh.nkb / S;
  const int nst = (kb1 - kb0 + KSUB - 1) / KSUB;            // stages of this CTA's k-range
  pdl_trigger();

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&maps.x);
    prefetch_tmap(&maps.w0);
    if (DUAL || sh.n1 < p.N) prefetch_tmap(&maps.w1);
    if (!DUAL && sh.n2 < p.N) prefetch_tmap(&maps.w2);
  }
  if (warp == 1) tmem_alloc(tmem_slot, sh.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // weight rows of this band: (map, first row) of its one or two boxes
      const CUtensorMap* wm0;
      const CUtensorMap* wm1 = &maps.w1;
      int wy;
      if (DUAL) {
        wm0 = &maps.w0;
        wy = band * (SW_BAND / 2);
      } else {
        const int n0 = band * SW_BAND;
        wm0 = n0 >= sh.n2 ? &maps.w2 : (n0 >= sh.n1 ? &maps.w1 : &maps.w0);
        wy = n0 >= sh.n2 ? n0 - sh.n2 : (n0 >= sh.n1 ? n0 - sh.n1 : n0);
      }
      auto nsub_of = [&](int j) { return min(KSUB, kb1 - (kb0 + j * KSUB)); };
      // weight sub-tiles of stage j into slot s
      auto load_w = [&](int s, int j) {
        for (int u = 0; u < nsub_of(j); ++u) {
          uint8_t* d = sW + (s * KSUB + u) * WSUB;
          const int x = (kb0 + j * KSUB + u) * SW_BK;
          tma_load_2d(d, wm0, x, wy, &full[s]);
          if (DUAL) tma_load_2d(d + (SW_BAND / 2) * 128, wm1, x, wy, &full[s]);
        }
      };
      auto stage_bytes = [&](int j) {
        return static_cast<uint32_t>(nsub_of(j) * (WSUB + X_BYTES));
      };
      const int npre = min(STAGES, nst);
      for (int j = 0; j < npre; ++j) {
        mbar_arrive_expect_tx(&full[j], stage_bytes(j));
        load_w(j, j);
      }
      pdl_wait();  // activations come from the previous kernel
      bool ok = true;
      int issued = 0;
      for (int j = 0; j < nst; ++j) {
        const int s = j % STAGES;
        const uint32_t ph = (j / STAGES) & 1;
        if (j >= npre) {
          if (!mbar_wait_ab(&empty[s], ph ^ 1, p.status, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], stage_bytes(j));
          load_w(s, j);
        }
        for (int u = 0; u < nsub_of(j); ++u)
          tma_load_2d(sX + (s * KSUB + u) * X_BYTES, &maps.x, (kb0 + j * KSUB + u) * SW_BK, row0, &full[s]);
        issued = j + 1;
      }
      // Do not go on while copies into this CTA's shared memory may be in flight.
      // (A stop can only come at a stage >= npre, so every pre-loaded stage also
      // had its activation tiles requested and is among the last `issued`.)
      if (!ok || *abort_flag) {
        for (int q = issued - 1; q >= 0 && q + STAGES >= issued; --q)
          mbar_wait(&full[q % STAGES], (q / STAGES) & 1, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(SW_BAND, sh.Mp);
      bool ok = true;
      for (int j = 0; j < nst; ++j) {
        const int s = j % STAGES;
        const uint32_t ph = (j / STAGES) & 1;
        if (!mbar_wait_ab(&full[s], ph, p.status, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int nsub = min(KSUB, kb1 - (kb0 + j * KSUB));
        for (int u = 0; u < nsub; ++u) {
          const uint32_t w_base = smem_u32(sW + (s * KSUB + u) * WSUB);
          const uint32_t x_base = smem_u32(sX + (s * KSUB + u) * X_BYTES);
#pragma unroll
          for (int k = 0; k < SW_BK / 16; ++k) {
            const uint32_t acc = (j > 0 || u > 0 || k > 0) ? 1u : 0u;
            tc_mma_bf16(tmem, sdesc_sw128(w_base + k * 32), sdesc_sw128(x_base + k * 32), idesc, acc);
          }
        }
        tc_commit(&empty[s]);
      }
      if (ok) tc_commit(acc_full);
    }
    __syncwarp();
  } else if (warp < 2 + SW_DRAIN_WARPS) {
    // TMEM lanes 32*(warp%4) .. +32 hold weight rows n of the band; column m is
    // activation row row0 + m.  Two warps per lane quarter take alternate
    // 16-column chunks.
    const int quad = warp & 3;
    const int h = (warp - 2) >> 2;
    const int n = quad * 32 + lane;
    const bool ok = __all_sync(0xffffffffu, mbar_wait_ab(acc_full, 0, p.status, abort_flag));
    if (ok) {
      tc_fence_after();
      fence_proxy_async_smem();  // the ring was last written by TMA, read by the MMAs
      const uint32_t tb = tmem + (static_cast<uint32_t>(quad * 32) << 16);
#pragma unroll 1
      for (int c = 16 * h; c < sh.Mp; c += 32) {
        uint32_t r[16];
        tmem_ld16(tb + c, r);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 16; ++e) red[(c + e) * SW_BAND + n] = __uint_as_float(r[e]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, sh.tmem_cols);
  }
  if (S > 1) cluster_sync_all();  // every CTA's partial is in its shared memory

  // ---- reduction over the cluster and epilogue: CTA `rank` finishes rows
  // [rank rows / S, (rank + 1) rows / S) of this block.
  pdl_wait();
  if (*abort_flag == 0) {
    uint32_t src[SW_MAX_CLUSTER];
    const uint32_t red_local = smem_u32(red);
#pragma unroll
    for (int c = 0; c < SW_MAX_CLUSTER; ++c) src[c] = c < S ? map_rank(red_local, c) : 0u;
    const int m_lo = rank * rows / S, m_hi = (rank + 1) * rows / S;
    if (S == 1)
      swap_epilogue<EPI, 2, true>(p, red, src, S, band, row0, m_lo, m_hi, warp, lane);
    else if (S <= 4)
      swap_epilogue<EPI, 2, false>(p, red, src, S, band, row0, m_lo, m_hi, warp, lane);
    else
      swap_epilogue<EPI, 1, false>(p, red, src, S, band, row0, m_lo, m_hi, warp, lane);
  }
  if (S > 1) cluster_sync_all();  // no CTA leaves while another still reads its partial
}

bool encode_sw(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint64_t row_elems,
               uint32_t box_rows) {
  EncodeTiledFn enc = get_encode_tiled();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_elems * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(SW_BK), box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                   box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

size_t smem_bytes(int wsub, int Mp, int stages, int ksub) {
  return static_cast<size_t>(stages) * ksub * (wsub + Mp * SW_BK * 2) + 1024 + 256;
}

template <int EPI>
cudaError_t ensure_attr() {
  static OncePerDevice once;
  return set_smem_limit_once(once, gemm_swap_kernel<EPI>, SW_RING_BUDGET + 1024 + 256);
}

cudaLaunchConfig_t make_cfg(dim3 grid, size_t smem, cudaStream_t s, cudaLaunchAttribute (&attr)[2],
                            int cluster) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(SW_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cfg;
}

// Clusters of `cluster` CTAs that fit on the device at once (cached per device and shape).
template <int EPI>
int max_clusters(int cluster, size_t smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, size_t>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, cluster, smem);
  std::lock_guard<std::mutex> lk(mu);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = make_cfg(dim3(cluster, 1, 1), smem, nullptr, attr, cluster);
  cfg.numAttrs = 1;  // the cluster dimension only
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, gemm_swap_kernel<EPI>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache[key] = n;
  return n;
}

template <int EPI>
cudaError_t run_swap(const void* A, int lda, const TcWeights& W, const GemmParams& p, cudaStream_t s) {
  cudaError_t e = ensure_attr<EPI>();
  if (e != cudaSuccess) return e;
  constexpr bool DUAL = EPI == kEpiSwiGLU;
  // row blocks of at most 256 rows, as even as 16-row granularity allows
  const int nrb = (p.M + kSwapRowBlock - 1) / kSwapRowBlock;
  const int per = (p.M + nrb - 1) / nrb;
  SwShape sh{};
  sh.Mp = (per + 15) / 16 * 16;
  const int nrb2 = (p.M + sh.Mp - 1) / sh.Mp;
  // A pass of the producer and MMA loops costs several hundred cycles whatever
  // a stage holds, so a stage takes as many 64-wide k-blocks (up to 4) as
  // still leaves two stages in the ring (a TMA probe on one SM streamed best
  // with about 100 KB per stage).
  const int kblock = SW_W_BYTES + sh.Mp * SW_BK * 2;
  sh.ksub = SW_RING_BUDGET / (2 * kblock);
  if (sh.ksub > 4) sh.ksub = 4;
  if (sh.ksub < 1) sh.ksub = 1;
  sh.stages = SW_RING_BUDGET / (sh.ksub * kblock);
  if (sh.stages > SW_MAX_STAGES) sh.stages = SW_MAX_STAGES;
  sh.nkb = p.K / SW_BK;
  sh.n1 = DUAL ? p.N : W.n1;
  sh.n2 = DUAL ? p.N : W.n2;
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(sh.Mp)) cols <<= 1;
  sh.tmem_cols = cols;
  const int bands = DUAL ? (p.N + SW_BAND / 2 - 1) / (SW_BAND / 2) : (p.N + SW_BAND - 1) / SW_BAND;
  const size_t smem = smem_bytes(SW_W_BYTES, sh.Mp, sh.stages, sh.ksub);

  // Cluster size: fewest k-blocks per CTA over the waves the clusters need,
  // with a wave's fixed work (launch, TMEM, cluster reduction, epilogue)
  // counted as a number of k-blocks.  Swept on GB300 over the 1B and 8B
  // projections of the accel-4 forwards (2, 6, 12, 24): 24 is best for the
  // RoPE epilogue (8B QKV at 192..316 rows 26.5 -> 20.1 us), 12 for the
  // residual one (8B O at 516..744 rows 49 -> 29..33 us), 2 for SwiGLU (whose
  // k-blocks carry twice the weights; larger values cost it 5-12%).
  const double wave_cost = EPI == kEpiRope ? 24.0 : (EPI == kEpiResid ? 12.0 : 2.0);
  const int units = bands * nrb2;
  int best = 1;
  double best_cost = 1e30;
  for (int S = 1; S <= SW_MAX_CLUSTER && S <= sh.nkb; ++S) {
    const int mc = max_clusters<EPI>(S, smem);
    if (mc <= 0) continue;
    const int waves = (units + mc - 1) / mc;
    const double cost = waves * (static_cast<double>((sh.nkb + S - 1) / S) + wave_cost);
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = S;
    }
  }

  SwMaps maps;
  memset(&maps, 0, sizeof(maps));
  if (!encode_sw(&maps.x, A, static_cast<uint64_t>(p.K), static_cast<uint64_t>(p.M),
                 static_cast<uint64_t>(lda), static_cast<uint32_t>(sh.Mp)))
    return cudaErrorInvalidValue;
  if (DUAL) {
    if (!encode_sw(&maps.w0, W.w0, p.K, p.N, p.K, SW_BAND / 2)) return cudaErrorInvalidValue;
    if (!encode_sw(&maps.w1, W.w1, p.K, p.N, p.K, SW_BAND / 2)) return cudaErrorInvalidValue;
  } else {
    const int r0 = W.n1 < p.N ? W.n1 : p.N;
    if (!encode_sw(&maps.w0, W.w0, p.K, r0, p.K, SW_BAND)) return cudaErrorInvalidValue;
    if (W.n1 < p.N) {
      const int r1 = (W.n2 < p.N ? W.n2 : p.N) - W.n1;
      if (!encode_sw(&maps.w1, W.w1, p.K, r1, p.K, SW_BAND)) return cudaErrorInvalidValue;
    }
    if (W.n2 < p.N) {
      if (!encode_sw(&maps.w2, W.w2, p.K, p.N - W.n2, p.K, SW_BAND)) return cudaErrorInvalidValue;
    }
  }
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = make_cfg(dim3(best, bands, nrb2), smem, s, attr, best);
  e = cudaLaunchKernelEx(&cfg, gemm_swap_kernel<EPI>, maps, sh, p);
  if (e != cudaSuccess) return e;
  if (p.launches) *p.launches += 1;
  return cudaSuccess;
}

bool aligned16(const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; }

}  // namespace

bool swap_supported(const void* A, int lda, const TcWeights& W, int epi, const GemmParams& p) {
  if (p.M <= kSkinnyMaxM || p.M > kSwapMaxM) return false;
  if (p.K % SW_BK != 0 || p.N % 16 != 0 || lda % 8 != 0 || p.ldo % 4 != 0) return false;
  if (!aligned16(A) || !aligned16(p.out)) return false;
  if (epi == kEpiResid && (p.resid == nullptr || !aligned16(p.resid))) return false;
  const void* ws[3] = {W.w0, W.w1, W.w2};
  for (const void* w : ws)
    if (!aligned16(w)) return false;
  if (epi != kEpiSwiGLU) {
    if (W.n1 < p.N && W.n1 % SW_BAND != 0) return false;
    if (W.n2 < p.N && W.n2 % SW_BAND != 0) return false;
  }
  if (epi == kEpiRope) {
    if (p.hd < 8 || p.hd % 8 != 0 || SW_BAND % p.hd != 0 || p.rope_cols % p.hd != 0) return false;
    if (p.pos == nullptr || p.cos_t == nullptr || p.sin_t == nullptr) return false;
  }
  return true;
}

bool swap_preferred(int epi, int M, int N, int K) {
  // Crossovers measured on GB300 for the Llama-3.2-1B and -8B projections
  // (CUDA-graph timed, weights streamed from HBM): above these row counts the
  // persistent tiled kernel keeps more SMs busy (SwiGLU needs two waves of
  // 128-row bands from 257 rows on) or streams its tiles faster.  Very wide
  // float32 outputs (LM heads, N >= 32768) stream their weights faster on the
  // tiled kernel at every row count (1B head at 40..456 rows: 0.68..0.94x).
  if (epi == kEpiStoreF32 && N >= 32768) return false;
  // Wide and deep weights (N, K >= 4096: every 8B projection) give the tiled
  // kernel at least 16 column tiles and 64 k-blocks per tile, and a third
  // 256-row block doubles the swapped kernel's weight passes: there the tiled
  // kernel wins from 268 rows (QKV + RoPE: 25.2 vs 25.7 us), 516 rows (O and
  // down + residual: 27.4 vs 28.9 us, 73.5 vs 92.3 us) and for SwiGLU at any
  // row count (20 rows: 45.9 vs 46.4 us; 220 rows: 56.7 vs 74.8 us).
  if (N >= 4096 && K >= 4096) {
    const int wide_limit = epi == kEpiSwiGLU ? 0 : (epi == kEpiResid ? 512 : 256);
    return M <= wide_limit;
  }
  const int limit = epi == kEpiSwiGLU ? 256 : (epi == kEpiResid ? 1024 : 768);
  return M <= limit;
}

cudaError_t launch_gemm_swap(const void* A, int lda, const TcWeights& W, int epi, const GemmParams& p,
                             cudaStream_t s) {
  switch (epi) {
    case kEpiStore: return run_swap<kEpiStore>(A, lda, W, p, s);
    case kEpiResid: return run_swap<kEpiResid>(A, lda, W, p, s);
    case kEpiSwiGLU: return run_swap<kEpiSwiGLU>(A, lda, W, p, s);
    case kEpiStoreF32: return run_swap<kEpiStoreF32>(A, lda, W, p, s);
    case kEpiRope: return run_swap<kEpiRope>(A, lda, W, p, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zsaa
