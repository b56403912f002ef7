// bf16 GEMM on the sm_103a tensor cores: out = epi(A[M,K] W[N,K]^T), fp32
// accumulation in tensor memory.
//
// Persistent kernels: one CTA per SM, or (gemm_pair_kernel, for many rows)
// one CTA pair per TPC on the 2-SM MMA.  Tiles are 128 x BN (tiles sharing a
// weight tile are adjacent, so weights stream from HBM once and are re-read
// from L2).  Whole waves of tiles are handed out round robin; with deep K the
// tiles of a ragged last wave may instead be cut into S aligned k-parts, dealt
// part-major so that the units of one round work on the same k-range of
// neighbouring tiles.  The non-final parts write fp32 partials (one slot each)
// and raise per-warp flags; the tile's last part waits (bounded) and adds them
// in part order before the epilogue -- deterministic, no extra launch, no
// atomics.
// Warp-specialised roles:
//   warp 0      TMA producer: 128B-swizzled A and W tiles (64 deep in K) into a
//               STAGES-deep shared-memory ring ("full" mbarriers, expect-tx);
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16)
//               into one of two TMEM accumulators and frees each stage with
//               tcgen05.commit on its "empty" mbarrier;
//   warps 2..5  epilogue: tcgen05.ld of the finished accumulator (one row per
//               thread), fused epilogue, 16-byte stores; then they hand the
//               accumulator back, so the next tile's MMAs overlap this epilogue.
// Epilogues: bf16 store; residual add (h += acc, in place); SwiGLU (the tile's
// first BN/2 accumulator columns are gate rows of W, the last BN/2 up rows of
// W2; out = silu(gate) * up); float32 store (logits); RoPE of the query/key
// heads at each row's original position, then bf16 store.
// Every mbarrier wait is bounded (2 s); on expiry the kernel sets the status
// word, the other roles stop waiting, in-flight copies are drained (bounded)
// and TMEM is freed before the CTA exits.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
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

// Work split: tiles [0, dp_tiles) go whole to unit t % units (whole waves).
// The tiles after them are split in k in one of two ways:
//   contiguous (sk_iters > 0): their sk_iters k-iterations are cut into
//     `units` equal contiguous ranges, across tile boundaries;
//   aligned (tail_R > 0): each of the tail_R tiles is cut into tail_S parts
//     of equal length (part s: k-blocks [s KB / S, (s + 1) KB / S)); part
//     q = s * tail_R + r (tile dp_tiles + r) goes to unit q % units, so the
//     units of a round work on the same k-part of neighbouring tiles.
// Tile t -> (m tile t % m_tiles, n tile t / m_tiles); the pair kernel's m
// tiles are 256 rows.
struct TileSched {
  int m_tiles, n_tiles, num_kb, total, dp_tiles;
  long long sk_iters;
  int tail_R, tail_S;
  float* ws;   // fp32 partials: one slot per contiguous unit or aligned non-final part
  int* flags;  // per slot, CTA of the unit and epilogue warp: 1 while the partial is ready
};

// One unit of work of a CTA: k-blocks [kb0, kb1) of a tile.
//   kind 0: the whole tile (epilogue directly);
//   kind 1: a non-final part of a split tile (write the partial to slot
//           `slot`, raise the flags);
//   kind 2: the final part of a split tile (add the `count` partials in
//           slots slot, slot + stride, ..., in that order; then the epilogue).
struct Item {
  int tile, kb0, kb1, kind, slot, count, stride;
};

// Work of unit `unit` of `units` (a CTA of the one-CTA kernel, a CTA pair of
// the pair kernel; both CTAs of a pair walk the same items).  Plain integer
// arithmetic, also run on the host to describe a plan (gemm_tc_schedule).
struct WorkIter {
  int t_dp, units, unit, q;
  long long it, end;
  __host__ __device__ __forceinline__ void init(const TileSched& ts, int u, int nunits) {
    t_dp = u;
    units = nunits;
    unit = u;
    q = u;
    const long long G = nunits;
    it = static_cast<long long>(u) * ts.sk_iters / G;
    end = static_cast<long long>(u + 1) * ts.sk_iters / G;
  }
  __host__ __device__ __forceinline__ bool next(const TileSched& ts, Item& w) {
    w.slot = 0;
    w.count = 0;
    w.stride = 1;
    if (t_dp < ts.dp_tiles) {
      w.tile = t_dp;
      w.kb0 = 0;
      w.kb1 = ts.num_kb;
      w.kind = 0;
      t_dp += units;
      return true;
    }
    const int KB = ts.num_kb;
    if (ts.sk_iters > 0) {
      if (it >= end) return false;
      const long long u = it / KB;
      const int a = static_cast<int>(it - u * KB);
      const long long rest = a + (end - it);
      const int b = static_cast<int>(rest < KB ? rest : KB);
      w.tile = ts.dp_tiles + static_cast<int>(u);
      w.kb0 = a;
      w.kb1 = b;
      if (a == 0 && b == KB) {
        w.kind = 0;
      } else if (a == 0) {
        // the tile's later parts are the first items of units unit+1 .. c_hi
        // (the unit holding iteration x is floor(((x + 1) * units - 1) / sk_iters))
        w.kind = 2;
        const long long G = units;
        const int c_hi = static_cast<int>(((u + 1) * KB * G - 1) / ts.sk_iters);
        w.slot = unit + 1;
        w.count = c_hi - unit;
      } else {
        w.kind = 1;
        w.slot = unit;
      }
      it += b - a;
      return true;
    }
    if (q >= ts.tail_R * ts.tail_S) return false;
    const int r = q % ts.tail_R, part = q / ts.tail_R, S = ts.tail_S;
    w.tile = ts.dp_tiles + r;
    w.kb0 = part * KB / S;
    w.kb1 = (part + 1) * KB / S;
    if (part == S - 1) {
      w.kind = 2;
      w.slot = r;  // parts 0 .. S-2 are in slots r, r + tail_R, ...
      w.count = S - 1;
      w.stride = ts.tail_R;
    } else {
      w.kind = 1;
      w.slot = q;
    }
    q += units;
    return true;
  }
};

// Bounded wait until a flag written by another CTA reads 1.
__device__ __forceinline__ bool wait_flag(const int* f, int* status, volatile int* abort) {
  unsigned long long t0 = 0;
  for (int n = 0;; ++n) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(f) : "memory");
    if (v == 1) return true;
    if ((n & 63) == 0) {
      if (*abort) return false;
      const unsigned long long t = globaltimer_ns();
      if (t0 == 0) t0 = t;
      else if (t - t0 > kWaitLimitNs) {
        if (status) atomicOr(status, kStatusTimeout);
        *abort = 1;
        return false;
      }
    }
  }
}

__device__ __forceinline__ float silu_f(float g) { return g / (1.f + __expf(-g)); }

__device__ __forceinline__ void store_bf16x16(bf16* dst, const float (&v)[16]) {
  uint32_t o[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) o[e] = pack_bf16x2(v[2 * e], v[2 * e + 1]);
  uint4* d = reinterpret_cast<uint4*>(dst);
  d[0] = make_uint4(o[0], o[1], o[2], o[3]);
  d[1] = make_uint4(o[4], o[5], o[6], o[7]);
}

// Adds the fp32 partials of `count` contributors (slot c at ws + c * cstride,
// column-major [BN][BM]: element (row, col) at slot[col * BM + row]) into this
// thread's row of the TMEM accumulator, contributor by contributor and column
// by column in increasing order, so each element is acc + p0 + p1 + ... in
// that order.  Every partial load is an L2 round trip, so the loads run two
// 32-column chunks ahead of the adds (a warp's loads of one column are one
// coalesced 128-byte line).
template <int BN>
__device__ __forceinline__ void fold_partials(uint32_t tbase, const float* ws, size_t cstride, int count,
                                              int rit) {
  constexpr int NCH = BN / 32;
  constexpr int DEPTH = NCH < 2 ? NCH : 2;
#pragma unroll 1
  for (int c = 0; c < count; ++c) {
    const float* slot = ws + static_cast<size_t>(c) * cstride + rit;
    float buf[DEPTH][32];
#pragma unroll
    for (int k = 0; k < DEPTH; ++k)
#pragma unroll
      for (int e = 0; e < 32; ++e) buf[k][e] = __ldcg(slot + static_cast<size_t>(32 * k + e) * BM);
#pragma unroll
    for (int ch = 0; ch < NCH; ++ch) {
      uint32_t r[32];
      __syncwarp();
      tmem_ld16(tbase + 32 * ch, *reinterpret_cast<uint32_t(*)[16]>(r));
      tmem_ld16(tbase + 32 * ch + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
      tmem_ld_wait();
#pragma unroll
      for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) + buf[ch % DEPTH][e]);
      tmem_st16(tbase + 32 * ch, *reinterpret_cast<const uint32_t(*)[16]>(r));
      tmem_st16(tbase + 32 * ch + 16, *reinterpret_cast<const uint32_t(*)[16]>(r + 16));
      if (ch + DEPTH < NCH) {
#pragma unroll
        for (int e = 0; e < 32; ++e)
          buf[ch % DEPTH][e] = __ldcg(slot + static_cast<size_t>(32 * (ch + DEPTH) + e) * BM);
      }
    }
    tmem_st_wait();  // this contributor's sums are in TMEM before the next pass reads them
  }
}

// Epilogue of one finished accumulator tile for this thread's row (any
// split-K partials are already folded into the accumulator).
template <int BN, int EPI>
__device__ __forceinline__ void tile_epilogue(uint32_t tbase, int row, bool row_ok, int n0,
                                              const GemmParams& p) {
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
        float gv[16], uv[16], v[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          gv[e] = __uint_as_float(g[e]);
          uv[e] = __uint_as_float(u[e]);
        }
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = silu_f(gv[e]) * uv[e];
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
          float v[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] = __uint_as_float(r[16 * h + e]);
          float4* dst = reinterpret_cast<float4*>(out + static_cast<size_t>(row) * p.ldo + n0 + c + 16 * h);
#pragma unroll
          for (int q = 0; q < 4; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
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
      float vss = 0.f;  // value heads: sum of squares of the stored (bf16) values
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
          float a1[16], a2[16], y1[16], y2[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            a1[e] = __uint_as_float(x1[e]);
            a2[e] = __uint_as_float(x2[e]);
          }
          if (rot) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float4 cs = cs4[q], sn = sn4[q];
              const float cv[4] = {cs.x, cs.y, cs.z, cs.w}, sv[4] = {sn.x, sn.y, sn.z, sn.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float a = a1[4 * q + e], b = a2[4 * q + e];
                y1[4 * q + e] = a * cv[e] - b * sv[e];
                y2[4 * q + e] = b * cv[e] + a * sv[e];
              }
            }
          } else {
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              y1[e] = a1[e];
              y2[e] = a2[e];
            }
          }
          bf16* rowp = out + static_cast<size_t>(row) * p.ldo + n0 + hs;
          store_bf16x16(rowp + c, y1);
          store_bf16x16(rowp + half + c, y2);
          if (!rot && p.vnorm_out != nullptr) {
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              const float r1 = __bfloat162float(__float2bfloat16_rn(y1[e]));
              const float r2 = __bfloat162float(__float2bfloat16_rn(y2[e]));
              vss += r1 * r1 + r2 * r2;
            }
          }
        }
      }
      if (!rot && p.vnorm_out != nullptr && row_ok && n0 + hs < p.N) {
        const int groups = (p.N - p.rope_cols) / hd;
        p.vnorm_out[static_cast<size_t>(row) * groups + (n0 + hs - p.rope_cols) / hd] = sqrtf(vss);
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

// Write this thread's row of the accumulator tile into the CTA's partial slot
// (column-major: element (row, col) at slot[col * BM + row]).
template <int BN>
__device__ __forceinline__ void write_partial(uint32_t tbase, float* slot, int rit) {
#pragma unroll 1
  for (int c = 0; c < BN; c += 32) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld16(tbase + c, *reinterpret_cast<uint32_t(*)[16]>(r));
    tmem_ld16(tbase + c + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
    tmem_ld_wait();
#pragma unroll
    for (int e = 0; e < 32; ++e) __stcg(slot + static_cast<size_t>(c + e) * BM + rit, __uint_as_float(r[e]));
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
  pdl_trigger();

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
      WorkIter wi;
      wi.init(ts, blockIdx.x, gridDim.x);
      // The weights are never written by another kernel: start streaming the
      // first stages' weight tiles before waiting for the previous kernel.
      int npre = 0;
      {
        WorkIter peek = wi;
        Item w0;
        if (peek.next(ts, w0)) {
          const int n0 = (w0.tile / ts.m_tiles) * BN;
          npre = min(C::STAGES, w0.kb1 - w0.kb0);
          for (int j = 0; j < npre; ++j) {
            const int kb = w0.kb0 + j;
            mbar_arrive_expect_tx(&full[j], C::STAGE_BYTES);
            if (EPI == kEpiSwiGLU) {
              tma_load_2d(sB + j * C::B_BYTES, &maps.b0, kb * BK, n0 / 2, &full[j]);
              tma_load_2d(sB + j * C::B_BYTES + (BN / 2) * 128, &maps.b1, kb * BK, n0 / 2, &full[j]);
            } else {
              const CUtensorMap* mb = n0 >= n2 ? &maps.b2 : (n0 >= n1 ? &maps.b1 : &maps.b0);
              const int nb = n0 >= n2 ? n0 - n2 : (n0 >= n1 ? n0 - n1 : n0);
              tma_load_2d(sB + j * C::B_BYTES, mb, kb * BK, nb, &full[j]);
            }
          }
        }
      }
      pdl_wait();
      Item w;
      while (ok && wi.next(ts, w)) {
        const int mt = w.tile % ts.m_tiles, nt = w.tile / ts.m_tiles;
        const int m0 = mt * BM, n0 = nt * BN;
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
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const int s = it % C::STAGES;
          const uint32_t ph = (it / C::STAGES) & 1;
          if (static_cast<int>(it) >= npre) {  // the first npre stages' weights are in flight already
            if (!mbar_wait_ab(&empty[s], ph ^ 1, p.status, abort_flag)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
            if (EPI == kEpiSwiGLU) {
              tma_load_2d(sB + s * C::B_BYTES, &maps.b0, kb * BK, n0 / 2, &full[s]);
              tma_load_2d(sB + s * C::B_BYTES + (BN / 2) * 128, &maps.b1, kb * BK, n0 / 2, &full[s]);
            } else {
              tma_load_2d(sB + s * C::B_BYTES, mb, kb * BK, nb, &full[s]);
            }
          }
          tma_load_2d(sA + s * C::A_BYTES, &maps.a, kb * BK, m0, &full[s]);
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
      WorkIter wi;
      wi.init(ts, blockIdx.x, gridDim.x);
      Item w;
      while (ok && wi.next(ts, w)) {
        const int ab = i & 1;
        const uint32_t use = static_cast<uint32_t>(i >> 1);
        ++i;
        if (!mbar_wait_ab(&acc_empty[ab], (use & 1) ^ 1, p.status, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(ab * BN);
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
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
                        (kb > w.kb0 || k > 0) ? 1u : 0u);
          tc_commit(&empty[s]);
        }
        tc_commit(&acc_full[ab]);
      }
    }
    __syncwarp();
  } else {
    // Epilogue: warp w reads TMEM lanes 32*(w%4) .. +32, i.e. tile rows.
    pdl_wait();
    const int quad = warp & 3;
    const int rit = quad * 32 + lane;  // row within the tile
    int i = 0;
    WorkIter wi;
    wi.init(ts, blockIdx.x, gridDim.x);
    Item w;
    while (wi.next(ts, w)) {
      const int mt = w.tile % ts.m_tiles, nt = w.tile / ts.m_tiles;
      const int row = mt * BM + rit;
      const int ab = i & 1;
      const uint32_t use = static_cast<uint32_t>(i >> 1);
      ++i;
      const bool ok = __all_sync(0xffffffffu, mbar_wait_ab(&acc_full[ab], use & 1, p.status, abort_flag));
      if (!ok) break;
      tc_fence_after();
      const uint32_t tbase = tmem + static_cast<uint32_t>(ab * BN) + (static_cast<uint32_t>(quad * 32) << 16);
      constexpr size_t kSlot = static_cast<size_t>(BM) * BN;
      if (w.kind == 1) {
        // a non-final k-part of a tail tile: its partial to slot w.slot
        write_partial<BN>(tbase, ts.ws + static_cast<size_t>(w.slot) * kSlot, rit);
        __threadfence();
        __syncwarp();
        if (lane == 0) {
          int* f = ts.flags + w.slot * 4 + quad;
          asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(f), "r"(1) : "memory");
        }
      } else {
        int c1 = -1;  // partials 0 .. c1 (none for a whole tile)
        if (w.kind == 2) {
          c1 = w.count - 1;
          bool got = true;
          for (int c = 0; c <= c1; ++c)
            got = got && wait_flag(ts.flags + (w.slot + c * w.stride) * 4 + quad, p.status, abort_flag);
          if (!__all_sync(0xffffffffu, got)) c1 = -1;  // gave up: status already set
        }
        if (c1 >= 0)
          fold_partials<BN>(tbase, ts.ws + static_cast<size_t>(w.slot) * kSlot, static_cast<size_t>(w.stride) * kSlot,
                            c1 + 1, rit);
        tile_epilogue<BN, EPI>(tbase, row, row < p.M, nt * BN, p);
        if (w.kind == 2) {
          __syncwarp();
          if (lane == 0)
            for (int c = 0; c <= c1; ++c) ts.flags[(w.slot + c * w.stride) * 4 + quad] = 0;
        }
      }
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

// ---------------------------------------------------------------------------
// CTA-pair kernel for many rows: tcgen05.mma.cta_group::2.
// A cluster of two CTAs (the two SMs of a TPC) computes 256 x 256 tiles.  CTA
// r of the pair stages A rows [m0 + 128 r, +128) and 128 of the tile's 256
// weight rows (rows n0 + 128 r; SwiGLU: CTA 0 the 128 gate rows of W, CTA 1 the
// same 128 up rows of W2) for each 64-deep k-block; the leader (rank 0) issues
// M=256, N=256 MMAs that read both CTAs' shared memory, and each CTA's TMEM
// receives its own 128 rows x 256 columns of the tile.  Per SM that is 32 KB of
// operands per 128 x 256 x 64 step instead of the one-CTA kernel's 48 KB, the
// stream that limits the one-CTA kernel at large M.
//   warp 0 (both CTAs)  TMA producer: this CTA's halves into a P_STAGES ring;
//                       the copies of both CTAs complete on the leader's
//                       "full" barrier, which the leader arms for both;
//   warp 1 (leader)     MMA issuer; tcgen05.commit multicasts each stage's
//                       release to both CTAs' "empty" barriers and each finished
//                       accumulator to both CTAs' "acc_full" barriers;
//   warps 2..5 (both)   epilogue of this CTA's 128 rows (the one-CTA kernel's),
//                       then release the accumulator on the leader's barrier.
// Work is split as in the one-CTA kernel, with the pair as the unit: whole
// tiles round robin (tile t -> row pair t % m_tiles, column tile t / m_tiles,
// so concurrent pairs share weight tiles in L2), then, for deep K, the
// k-iterations of the last tiles in equal ranges; CTA r of a pair that holds
// a later part of a split tile writes its 128 rows of the partial to slot
// blockIdx.x, and CTA r of the tile's first pair P adds the slots 2c + r of the
// contributing pairs c, in pair order.
// Every wait is bounded; a CTA that gives up waits briefly for its own copies
// in flight and still reaches the closing cluster barrier.
constexpr int P_BN = 256;
constexpr int P_STAGES = 6;
constexpr int P_A_BYTES = BM * BK * 2;          // this CTA's 128 rows of A
constexpr int P_B_BYTES = (P_BN / 2) * BK * 2;  // this CTA's 128 weight rows
constexpr int P_STAGE_BYTES = P_A_BYTES + P_B_BYTES;
constexpr size_t P_SMEM = static_cast<size_t>(P_STAGES) * P_STAGE_BYTES + 1024 + 256;
constexpr uint32_t P_TMEM_COLS = 2 * P_BN;  // two accumulators
constexpr double kPairTileCost = 0.9;
// K of at least this many 64-deep k-blocks counts as deep in the tile plan.
constexpr int kDeepKb = 64;
// From this many k-blocks on (the 8B down projection, 224) a ragged last wave
// may be cut into aligned k-parts; below it (1B down, 128; 64) the contiguous
// stream-K split measured better, or no split at all.
constexpr int kVeryDeepKb = 192;

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_pair_kernel(const __grid_constant__ TcMaps maps, const int n1, const int n2,
                     const GemmParams p, const TileSched ts) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + P_STAGES * P_A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + P_STAGES * P_STAGE_BYTES);
  uint64_t* empty = full + P_STAGES;
  uint64_t* acc_full = empty + P_STAGES;  // [2]
  uint64_t* acc_empty = acc_full + 2;     // [2], used in the leader
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = static_cast<int>(cluster_rank());
  const int pair = static_cast<int>(blockIdx.x >> 1), npairs = static_cast<int>(gridDim.x >> 1);
  pdl_trigger();

  if (threadIdx.x == 0) {
    for (int s = 0; s < P_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 8);  // four epilogue warps in each CTA
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
  if (warp == 1) tmem_alloc_pair(tmem_slot, P_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised before any copy or arrival crosses
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      const uint32_t full_leader = map_rank(smem_u32(full), 0);
      // this CTA's 128 weight rows of column tile nt: (map, first row)
      auto w_rows = [&](int nt, const CUtensorMap*& mb, int& wy) {
        const int n0 = nt * P_BN;
        if (EPI == kEpiSwiGLU) {
          mb = rank == 0 ? &maps.b0 : &maps.b1;
          wy = n0 / 2;
        } else {
          mb = n0 >= n2 ? &maps.b2 : (n0 >= n1 ? &maps.b1 : &maps.b0);
          wy = (n0 >= n2 ? n0 - n2 : (n0 >= n1 ? n0 - n1 : n0)) + rank * (P_BN / 2);
        }
      };
      uint32_t it = 0, issued = 0;
      bool ok = true;
      WorkIter wi;
      wi.init(ts, pair, npairs);
      // weights are never written by another kernel: request the first item's
      // first stages before waiting for the previous kernel
      int npre = 0;
      {
        WorkIter peek = wi;
        Item w0;
        if (peek.next(ts, w0)) {
          const CUtensorMap* mb;
          int wy;
          w_rows(w0.tile / ts.m_tiles, mb, wy);
          npre = min(P_STAGES, w0.kb1 - w0.kb0);
          for (int j = 0; j < npre; ++j) {
            if (rank == 0) mbar_arrive_expect_tx(&full[j], 2 * P_STAGE_BYTES);
            tma_load_2d_pair(sB + j * P_B_BYTES, mb, (w0.kb0 + j) * BK, wy, full_leader + 8u * j);
          }
        }
      }
      pdl_wait();
      Item w;
      while (ok && wi.next(ts, w)) {
        const int mp = w.tile % ts.m_tiles, nt = w.tile / ts.m_tiles;
        const int m0 = mp * (2 * BM) + rank * BM;
        const CUtensorMap* mb;
        int wy;
        w_rows(nt, mb, wy);
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const int s = it % P_STAGES;
          const uint32_t ph = (it / P_STAGES) & 1;
          if (static_cast<int>(it) >= npre) {
            if (!mbar_wait_ab(&empty[s], ph ^ 1, p.status, abort_flag)) {
              ok = false;
              break;
            }
            if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * P_STAGE_BYTES);
            tma_load_2d_pair(sB + s * P_B_BYTES, mb, kb * BK, wy, full_leader + 8u * s);
          }
          tma_load_2d_pair(sA + s * P_A_BYTES, &maps.a, kb * BK, m0, full_leader + 8u * s);
          issued = it + 1;
        }
      }
      // The copies land on the leader's barrier, which this thread cannot always
      // watch: after a stop, give copies still in flight time to land (a TMA
      // copy takes microseconds) before the CTA can exit.
      if ((!ok || *abort_flag) && issued > 0) {
        const unsigned long long t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 200000ull) __nanosleep(1000);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(2 * BM, P_BN);
      uint32_t it = 0;
      bool ok = true;
      int i = 0;
      WorkIter wi;
      wi.init(ts, pair, npairs);
      Item w;
      while (ok && wi.next(ts, w)) {
        const int ab = i & 1;
        const uint32_t use = static_cast<uint32_t>(i >> 1);
        ++i;
        if (!mbar_wait_cluster_ab(&acc_empty[ab], (use & 1) ^ 1, p.status, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(ab * P_BN);
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const int s = it % P_STAGES;
          const uint32_t ph = (it / P_STAGES) & 1;
          if (!mbar_wait_ab(&full[s], ph, p.status, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(sA + s * P_A_BYTES);
          const uint32_t b_base = smem_u32(sB + s * P_B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma_bf16_pair(d_tmem, sdesc_sw128(a_base + k * 32), sdesc_sw128(b_base + k * 32), idesc,
                             (kb > w.kb0 || k > 0) ? 1u : 0u);
          tc_commit_pair(&empty[s]);
        }
        if (ok) tc_commit_pair(&acc_full[ab]);
      }
    }
    __syncwarp();
  } else {
    // Epilogue: warp w reads TMEM lanes 32*(w%4) .. +32 -- this CTA's tile rows.
    pdl_wait();
    const int quad = warp & 3;
    const int rit = quad * 32 + lane;
    const uint32_t acc_empty_leader = map_rank(smem_u32(acc_empty), 0);
    constexpr size_t kSlot = static_cast<size_t>(BM) * P_BN;  // one CTA's partial
    int i = 0;
    WorkIter wi;
    wi.init(ts, pair, npairs);
    Item w;
    while (wi.next(ts, w)) {
      const int mp = w.tile % ts.m_tiles, nt = w.tile / ts.m_tiles;
      const int row = mp * (2 * BM) + rank * BM + rit;
      const int ab = i & 1;
      const uint32_t use = static_cast<uint32_t>(i >> 1);
      ++i;
      const bool ok = __all_sync(0xffffffffu, mbar_wait_ab(&acc_full[ab], use & 1, p.status, abort_flag));
      if (!ok) break;
      tc_fence_after();
      const uint32_t tbase = tmem + static_cast<uint32_t>(ab * P_BN) + (static_cast<uint32_t>(quad * 32) << 16);
      // a pair's slot q holds CTA r's 128 rows at CTA slot 2q + r
      if (w.kind == 1) {
        // a non-final k-part of a tail tile: this CTA's rows to its slot
        write_partial<P_BN>(tbase, ts.ws + static_cast<size_t>(2 * w.slot + rank) * kSlot, rit);
        __threadfence();
        __syncwarp();
        if (lane == 0) {
          int* f = ts.flags + (2 * w.slot + rank) * 4 + quad;
          asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(f), "r"(1) : "memory");
        }
      } else {
        int c1 = -1;  // partials 0 .. c1 (none for a whole tile)
        if (w.kind == 2) {
          c1 = w.count - 1;
          bool got = true;
          for (int c = 0; c <= c1; ++c)
            got = got && wait_flag(ts.flags + (2 * (w.slot + c * w.stride) + rank) * 4 + quad, p.status, abort_flag);
          if (!__all_sync(0xffffffffu, got)) c1 = -1;  // gave up: status already set
        }
        if (c1 >= 0)
          fold_partials<P_BN>(tbase, ts.ws + static_cast<size_t>(2 * w.slot + rank) * kSlot,
                              2 * static_cast<size_t>(w.stride) * kSlot, c1 + 1, rit);
        tile_epilogue<P_BN, EPI>(tbase, row, row < p.M, nt * P_BN, p);
        if (w.kind == 2) {
          __syncwarp();
          if (lane == 0)
            for (int c = 0; c <= c1; ++c) ts.flags[(2 * (w.slot + c * w.stride) + rank) * 4 + quad] = 0;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc_empty_leader + 8u * ab);
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no copy, commit or arrival of this tile loop still targets the other CTA
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, P_TMEM_COLS);
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
                   int grid, cudaStream_t s) {
  using C = TcCfg<BN>;
  static OncePerDevice once;
  const cudaError_t attr_err = set_smem_limit_once(once, gemm_tc_kernel<BN, EPI>, static_cast<int>(C::SMEM));
  if (attr_err != cudaSuccess) return attr_err;
  ZSAA_LAUNCH(gemm_tc_kernel<BN, EPI>, dim3(grid), dim3(kThreads), C::SMEM, s, maps, n1, n2, p, ts);
  if (p.launches) *p.launches += 1;
  return cudaGetLastError();
}

template <int BN>
cudaError_t dispatch_epi(int epi, const TcMaps& maps, int n1, int n2, const GemmParams& p,
                         const TileSched& ts, int grid, cudaStream_t s) {
  switch (epi) {
    case kEpiStore: return run_tc<BN, kEpiStore>(maps, n1, n2, p, ts, grid, s);
    case kEpiResid: return run_tc<BN, kEpiResid>(maps, n1, n2, p, ts, grid, s);
    case kEpiSwiGLU: return run_tc<BN, kEpiSwiGLU>(maps, n1, n2, p, ts, grid, s);
    case kEpiStoreF32: return run_tc<BN, kEpiStoreF32>(maps, n1, n2, p, ts, grid, s);
    case kEpiRope: return run_tc<BN, kEpiRope>(maps, n1, n2, p, ts, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

template <int EPI>
cudaError_t pair_attr() {
  static OncePerDevice once;
  return set_smem_limit_once(once, gemm_pair_kernel<EPI>, static_cast<int>(P_SMEM));
}

cudaLaunchConfig_t pair_cfg(int pairs, cudaStream_t s, cudaLaunchAttribute (&attr)[2]) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * pairs);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = P_SMEM;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cfg;
}

// CTA pairs of the pair kernel resident at once (0 if the query fails), per device.
template <int EPI>
int pair_slots() {
  static std::mutex mu;
  static int cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  std::lock_guard<std::mutex> lk(mu);
  if (cached[dev] != 0) return cached[dev] > 0 ? cached[dev] : 0;
  int n = 0;
  if (pair_attr<EPI>() == cudaSuccess) {
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = pair_cfg(1, nullptr, attr);
    cfg.numAttrs = 1;  // the cluster dimension only
    if (cudaOccupancyMaxActiveClusters(&n, gemm_pair_kernel<EPI>, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();
  cached[dev] = n > 0 ? n : -1;
  return n > 0 ? n : 0;
}

// ZSAA_GEMM_PAIRS=0 in the environment (read once per process) keeps every
// tiled GEMM on one CTA: a diagnostic switch, so the one-CTA kernel's whole
// and split paths -- the fallback where CTA pairs cannot be scheduled -- can
// be tested and timed against the pairs on a GPU that has them.
bool pairs_enabled() {
  static const bool on = [] {
    const char* e = std::getenv("ZSAA_GEMM_PAIRS");
    return !(e != nullptr && e[0] == '0');
  }();
  return on;
}

int pair_slots_for(int epi) {
  switch (epi) {
    case kEpiStore: return pair_slots<kEpiStore>();
    case kEpiResid: return pair_slots<kEpiResid>();
    case kEpiSwiGLU: return pair_slots<kEpiSwiGLU>();
    case kEpiStoreF32: return pair_slots<kEpiStoreF32>();
    case kEpiRope: return pair_slots<kEpiRope>();
    default: return 0;
  }
}

template <int EPI>
cudaError_t run_pair(const TcMaps& maps, int n1, int n2, const GemmParams& p, const TileSched& ps,
                     int pairs, cudaStream_t s) {
  cudaError_t e = pair_attr<EPI>();
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = pair_cfg(pairs, s, attr);
  e = cudaLaunchKernelEx(&cfg, gemm_pair_kernel<EPI>, maps, n1, n2, p, ps);
  if (e != cudaSuccess) return e;
  if (p.launches) *p.launches += 1;
  return cudaSuccess;
}

cudaError_t dispatch_pair(int epi, const TcMaps& maps, int n1, int n2, const GemmParams& p,
                          const TileSched& ps, int pairs, cudaStream_t s) {
  switch (epi) {
    case kEpiStore: return run_pair<kEpiStore>(maps, n1, n2, p, ps, pairs, s);
    case kEpiResid: return run_pair<kEpiResid>(maps, n1, n2, p, ps, pairs, s);
    case kEpiSwiGLU: return run_pair<kEpiSwiGLU>(maps, n1, n2, p, ps, pairs, s);
    case kEpiStoreF32: return run_pair<kEpiStoreF32>(maps, n1, n2, p, ps, pairs, s);
    case kEpiRope: return run_pair<kEpiRope>(maps, n1, n2, p, ps, pairs, s);
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

// Whether to cut the ragged last wave of a plan into aligned k-parts, from a
// model fitted to GB300 measurements of forced plans on the 8B projections
// (graph-timed, weights from HBM): with Tw the time of one full wave,
//   whole: W Tw + Tw min(1, 0.25 + 4 R / units)  (only a nearly empty last
//          wave runs faster: 8B down at 1204 rows spent about 25 us on its
//          last 4 of 76 pair tiles, but 70-73 us on 20, 36 or 52 of them,
//          as on a full wave);
//   split: W Tw + Tw / S + 8 us + 5.5 us (S - 1), all R S parts in one round
//          (one partial written, S - 1 read back by the tile's last part:
//          17-31 us measured at S = 3..5 on 224 k-blocks; two rounds measured
//          slower than predicted).
// So the split pays only on deep K (8B down: 1536 rows 145.5 -> 114.3 us,
// 5084 rows 397.2 -> 364.2 us); on 64 k-blocks it measured 3-37% slower.
struct TailPlan {
  int S;  // k-parts per remainder tile; 1: whole tiles only
};
TailPlan tail_plan(int total, int units, int kb, double step_us, bool can_split, int max_slots) {
  const int W = total / units, R = total - W * units;
  TailPlan tp{1};
  if (!can_split || R == 0 || kb < kDeepKb) return tp;
  const double tw = kb * step_us;
  double best = tw * std::min(1.0, 0.25 + 4.0 * R / units);
  for (int S = 2; S <= 8; ++S) {
    if (kb / S < 8 || R * (S - 1) > max_slots || R * S > units) break;
    const double t = tw / S + 8.0 + 5.5 * (S - 1);
    if (t < best - 1e-9) {
      best = t;
      tp.S = S;
    }
  }
  return tp;
}

// Fill t's work split from tail_plan; returns the grid in units.
int apply_tail(TileSched& t, int units, const TailPlan& tp) {
  t.sk_iters = 0;
  if (tp.S <= 1) {
    t.dp_tiles = t.total;
    t.tail_R = 0;
    t.tail_S = 1;
    return t.total < units ? t.total : units;
  }
  const int W = t.total / units;
  t.dp_tiles = W * units;
  t.tail_R = t.total - t.dp_tiles;
  t.tail_S = tp.S;
  const int parts = t.tail_R * tp.S;
  return W > 0 ? units : (parts < units ? parts : units);
}

// What the tile plan needs besides the call's shape: how many CTAs (one per
// SM) and CTA pairs the device runs at once for this epilogue, the split-K
// workspace, and which tile widths the weight splits and RoPE heads allow.
struct TilePlanIn {
  int epi, M, N, K;
  int sms;         // one-CTA kernel: CTAs resident at once
  int slots;       // pair kernel: CTA pairs resident at once; 0: no pairs
  bool can_split;  // a split-K workspace and flags were given
  int cta_slots;   // its partial slots (BM x 256 fp32, four flags each)
  bool bn64, bn128, bn256;
  bool width_ok(int BN) const { return BN == 64 ? bn64 : (BN == 128 ? bn128 : (BN == 256 && bn256)); }
};

// The plan: the one-CTA kernel's tile width, grid and work split, and, when
// pairs > 0, the CTA-pair kernel's (which then runs instead).  The splits'
// workspace pointers are left to the caller.
struct TilePlanOut {
  int BN, grid;
  TileSched ts;
  int pairs;
  TileSched ps;
};

// Host only: no device calls.  False when no tile width fits.
bool plan_tiles(const TilePlanIn& in, TilePlanOut& o) {
  const int epi = in.epi, sms = in.sms, slots = in.slots, cta_slots = in.cta_slots;
  const bool can_split = in.can_split;
  const int vn = epi == kEpiSwiGLU ? 2 * in.N : in.N;
  const int m_tiles = (in.M + BM - 1) / BM;
  const int num_kb = in.K / BK;
  int BN = 0;
  bool plan_pairs = false;
  TailPlan plan_tp{1};
  if (num_kb >= kDeepKb) {
    // Deep K (>= 64 k-blocks: every 8B projection, the 1B down projection):
    // the plan with the least waves x cost of one k-block step
    // -- one-CTA tiles 128 or 256 wide, or 256 x 256 tiles on CTA pairs (only
    // with two or more 128-row tiles: a lone one would leave half of each pair
    // tile empty); then its ragged last wave possibly cut into aligned k-parts
    // (tail_plan).  The step costs are GB300 graph-timed averages over the 1B
    // and 8B pruned-forward shapes with every SM streaming: 0.27 us (128-wide)
    // and 0.36 us (256-wide) per 64-deep k-block, 0.34 us per pair step.
    // Narrow tiles win only while they still fit one wave (8B QKV at 316
    // rows: 25.2 us against 30.1 on pairs); pairs win while they add no wave
    // (8B O at 744 rows: 27.7 us against 33.0 on the swapped kernel).
    double best = 1e30;
    int best_tiles = 0;
    for (int cand : {128, 256}) {
      if (!in.width_ok(cand)) continue;
      const int tiles = m_tiles * ((vn + cand - 1) / cand);
      const double cost = static_cast<double>((tiles + sms - 1) / sms) * (cand == 256 ? 0.36 : 0.27);
      if (cost < best - 1e-9) {
        best = cost;
        BN = cand;
        best_tiles = tiles;
      }
    }
    if (slots > 0 && m_tiles >= 2) {
      const int ptiles = ((m_tiles + 1) / 2) * ((vn + P_BN - 1) / P_BN);
      const double cost = static_cast<double>((ptiles + slots - 1) / slots) * 0.34;
      if (cost < best - 1e-9) {
        BN = P_BN;
        plan_pairs = true;
        best_tiles = ptiles;
      }
    }
    if (BN != 0 && num_kb >= kVeryDeepKb) {
      plan_tp = plan_pairs ? tail_plan(best_tiles, slots, num_kb, 0.34, can_split && 2 * slots <= kMaxGemmCtas,
                                       cta_slots / 2)
                           : tail_plan(best_tiles, sms, num_kb, BN == 256 ? 0.36 : 0.27,
                                       can_split && sms <= kMaxGemmCtas, cta_slots);
    }
  }
  if (BN == 0) {
    // Tile width by problem size, from sweeps of the pruned-prefill shapes on
    // GB300 (graph-timed): narrow tiles only while M is small enough that wide
    // ones leave most SMs idle; the SwiGLU GEMM (2x the columns) always wide.
    // (also wide whenever there are two waves of wide tiles: the LM head's
    // 128256 columns would otherwise re-read the activation thousands of times)
    const long wide_tiles = static_cast<long>(m_tiles) * ((vn + 255) / 256);
    const int want = (epi == kEpiSwiGLU || wide_tiles >= 2L * sms)
                         ? 256
                         : (in.M <= 256 ? 64 : (in.M <= 768 ? 128 : 256));
    for (int cand : {64, 128, 256})
      if (in.width_ok(cand) && (BN == 0 || cand <= want)) BN = cand;
    if (BN == 0) return false;
  }
  TileSched ts{};
  ts.m_tiles = m_tiles;
  ts.n_tiles = (vn + BN - 1) / BN;
  ts.num_kb = num_kb;
  ts.total = ts.m_tiles * ts.n_tiles;
  // Whole tiles, except with deep K and a ragged last wave:
  //  - very deep K, where tail_plan found it cheaper: the last wave's tiles cut
  //    into aligned k-parts (8B down at 1536 rows 145.5 -> 114.3 us, at 6456
  //    rows 499.7 -> 461.3 us, against the rules below);
  //  - else, from two waves on, stream-K over the last one-to-two waves (or
  //    over everything, for problems smaller than two waves). Measured on
  //    GB300: the contiguous split pays at 128 and 224 k-blocks from a quarter
  //    of the last wave's SM-time idle (8B down at 1196 rows: 99.2 us split
  //    against 140.3 whole), but at 64 k-blocks only from 40% idle (8B QKV
  //    at 1732 rows, 26% idle: 79.3 split against 65.3 whole; 8B O at 1204
  //    rows, 47% idle: 43.5 against 46.7), and never within one wave, where it
  //    only adds the partial hand-off (8B down at 744 rows: 81.5 against 74.6).
  const double split_idle = num_kb >= 2 * kDeepKb ? 0.25 : 0.40;
  int grid;
  if (!plan_pairs && plan_tp.S > 1) {
    grid = apply_tail(ts, sms, plan_tp);
  } else {
    ts.tail_R = 0;
    ts.tail_S = 1;
    const int waves = (ts.total + sms - 1) / sms;
    const double idle = 1.0 - static_cast<double>(ts.total) / (static_cast<double>(waves) * sms);
    const bool split_ok = can_split && sms <= kMaxGemmCtas && sms <= cta_slots;
    if (plan_pairs || !split_ok || num_kb < kDeepKb || waves < 2 || idle <= split_idle) {
      ts.dp_tiles = ts.total;
      ts.sk_iters = 0;
      grid = ts.total < sms ? ts.total : sms;
    } else {
      ts.dp_tiles = ts.total >= 2 * sms ? (ts.total / sms - 1) * sms : 0;
      ts.sk_iters = static_cast<long long>(ts.total - ts.dp_tiles) * ts.num_kb;
      grid = sms;
      if (ts.dp_tiles == 0) {  // small problem: keep at least 8 k-blocks per CTA
        const long long g = ts.sk_iters / 8;
        grid = static_cast<int>(g < 1 ? 1 : (g < sms ? g : sms));
      }
    }
  }
  // CTA pairs (256 x 256 tiles on the 2-SM MMA): per MMA step each SM streams
  // 32 KB of operands instead of 48 KB, the stream that limits the one-CTA
  // kernel at many rows.  With deep K the plan above decides; otherwise
  // (measured on the Llama-3.2-1B projections at K = 2048, 288..4096 rows) a
  // pair wave takes 0.84..0.96 of a one-CTA wave, but pairing 128-row tiles
  // can leave half a pair empty and add a wave, and in a single short-K wave
  // the pair's extra synchronisation costs 1..4%, so pairs are taken when they
  // save waves at kPairTileCost each.
  TileSched ps{};
  int pairs = 0;
  if (BN == P_BN && slots > 0) {
    ps.m_tiles = (m_tiles + 1) / 2;  // 256-row tiles
    ps.n_tiles = ts.n_tiles;
    ps.num_kb = ts.num_kb;
    ps.total = ps.m_tiles * ps.n_tiles;
    ps.tail_R = 0;
    ps.tail_S = 1;
    const int waves_pair = (ps.total + slots - 1) / slots;
    const double pair_idle = 1.0 - static_cast<double>(ps.total) / (static_cast<double>(waves_pair) * slots);
    const bool pair_split_ok = can_split && 2 * slots <= kMaxGemmCtas && 2 * slots <= cta_slots;
    if (plan_pairs && plan_tp.S > 1) {
      pairs = apply_tail(ps, slots, plan_tp);
    } else if (plan_pairs && pair_split_ok && waves_pair >= 2 && pair_idle > split_idle) {
      // deep K with a ragged last wave: the contiguous stream-K split over the pairs
      pairs = slots;
      ps.dp_tiles = ps.total >= 2 * pairs ? (ps.total / pairs - 1) * pairs : 0;
      ps.sk_iters = static_cast<long long>(ps.total - ps.dp_tiles) * ps.num_kb;
      if (ps.dp_tiles == 0) {  // small problem: keep at least 8 k-blocks per pair
        const long long g = ps.sk_iters / 8;
        pairs = static_cast<int>(g < 1 ? 1 : (g < slots ? g : slots));
      }
    } else if (plan_pairs) {
      pairs = apply_tail(ps, slots, TailPlan{1});
    } else if (num_kb < kDeepKb) {
      const int waves_one = (ts.total + sms - 1) / sms;
      if (waves_pair * kPairTileCost < waves_one && waves_one >= 2) pairs = apply_tail(ps, slots, TailPlan{1});
    }
  }
  o.BN = BN;
  o.grid = grid;
  o.ts = ts;
  o.pairs = pairs;
  o.ps = ps;
  return true;
}

}  // namespace

cudaError_t launch_gemm_tc(const void* A, int lda, const TcWeights& W, int epi,
                           const GemmParams& p, cudaStream_t s) {
  if (p.K % BK != 0 || p.N % 16 != 0 || lda % 8 != 0) return cudaErrorInvalidValue;
  // a handful of rows: 128-row tiles would idle most of the tensor core and
  // most SMs; stream the weights instead
  if (skinny_supported(A, lda, W, epi, p)) return launch_gemm_skinny(A, lda, W, epi, p, s);
  // a few hundred rows: weight band as the 128-row operand, K split over a cluster
  if (swap_preferred(epi, p.M, p.N, p.K) && swap_supported(A, lda, W, epi, p))
    return launch_gemm_swap(A, lda, W, epi, p, s);
  const int vn = epi == kEpiSwiGLU ? 2 * p.N : p.N;
  TilePlanIn in;
  in.epi = epi;
  in.M = p.M;
  in.N = p.N;
  in.K = p.K;
  in.sms = num_sms();
  in.slots = (pairs_enabled() && bn_ok(P_BN, epi, W, p)) ? pair_slots_for(epi) : 0;
  // Split-K workspace: slots of BM x 256 fp32 per CTA, four flags each.
  in.can_split = p.splitk_ws != nullptr && p.splitk_flags != nullptr;
  in.cta_slots = in.can_split ? static_cast<int>(std::min<size_t>(p.splitk_ws_elems / (static_cast<size_t>(BM) * 256),
                                                                   kSplitKFlags / 4))
                              : 0;
  in.bn64 = bn_ok(64, epi, W, p);
  in.bn128 = bn_ok(128, epi, W, p);
  in.bn256 = bn_ok(256, epi, W, p);
  TilePlanOut pl;
  if (!plan_tiles(in, pl)) return cudaErrorInvalidValue;
  const int BN = pl.BN, grid = pl.grid, pairs = pl.pairs;
  TileSched ts = pl.ts, ps = pl.ps;
  ts.ws = ps.ws = p.splitk_ws;
  ts.flags = ps.flags = p.splitk_flags;
  TcMaps maps;
  memset(&maps, 0, sizeof(maps));
  const uint32_t brows = (pairs > 0 || epi == kEpiSwiGLU) ? BN / 2 : BN;
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
  if (pairs > 0) return dispatch_pair(epi, maps, n1, n2, p, ps, pairs, s);
  switch (BN) {
    case 256: return dispatch_epi<256>(epi, maps, n1, n2, p, ts, grid, s);
    case 128: return dispatch_epi<128>(epi, maps, n1, n2, p, ts, grid, s);
    default: return dispatch_epi<64>(epi, maps, n1, n2, p, ts, grid, s);
  }
}

int gemm_tc_schedule(int epi, int M, int N, int K, int hd, int sms, int pair_slots, int split_slots,
                     int* plan, int* items, long long cap, long long* n_items) {
  TilePlanIn in;
  in.epi = epi;
  in.M = M;
  in.N = N;
  in.K = K;
  in.sms = sms;
  // one weight matrix (no weight splits); RoPE heads of hd dims in every column tile
  auto width_ok = [&](int BN) { return epi != kEpiRope || BN % hd == 0; };
  in.slots = width_ok(P_BN) ? pair_slots : 0;
  in.can_split = split_slots > 0;
  in.cta_slots = in.can_split ? std::min(split_slots, static_cast<int>(kSplitKFlags / 4)) : 0;
  in.bn64 = width_ok(64);
  in.bn128 = width_ok(128);
  in.bn256 = width_ok(256);
  TilePlanOut pl;
  if (!plan_tiles(in, pl)) return -1;
  const bool pairs = pl.pairs > 0;
  const TileSched& ts = pairs ? pl.ps : pl.ts;
  const int units = pairs ? pl.pairs : pl.grid;
  if (ts.sk_iters > 0x7fffffffLL) return -1;
  const int fields[12] = {pl.BN, pairs ? 1 : 0, units, ts.m_tiles, ts.n_tiles, ts.num_kb, ts.total,
                          ts.dp_tiles, static_cast<int>(ts.sk_iters), ts.tail_R, ts.tail_S, 0};
  for (int i = 0; i < 12; ++i) plan[i] = fields[i];
  // every item of a sound plan covers at least one k-block: more items than
  // tile k-blocks means a unit's iterator does not advance
  const long long limit = static_cast<long long>(ts.total) * ts.num_kb;
  long long n = 0;
  for (int u = 0; u < units; ++u) {
    WorkIter it;
    it.init(ts, u, units);
    Item w;
    while (it.next(ts, w)) {
      if (n >= limit) return -2;
      if (items != nullptr && n < cap) {
        int* o = items + 8 * n;
        o[0] = u;
        o[1] = w.tile;
        o[2] = w.kb0;
        o[3] = w.kb1;
        o[4] = w.kind;
        o[5] = w.slot;
        o[6] = w.count;
        o[7] = w.stride;
      }
      ++n;
    }
  }
  *n_items = n;
  return 0;
}

}  // namespace zsaa
