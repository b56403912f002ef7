// Causal (or bidirectional) grouped-query attention, Eq. 1, on the sm_103a
// tensor cores, for bf16 heads of 64 or 128 dims (HD).
//
// Persistent: one CTA per SM walks work items (query block of 128 rows, query
// head, sequence; longest first) and streams their key blocks through one
// pipeline, so TMA, MMA and softmax of consecutive items overlap.  For every
// key block of BN (128 keys for HD = 64, 64 for HD = 128, so that both fit the
// same shared-memory ring; causal: up to the diagonal):
//   MMA1  S = Q K^T          (tcgen05, M = 128 queries, N = BN keys, K = HD) -> TMEM
//   softmax warps (one query row per thread, TMEM lane = row): scale, mask,
//         running max m and sum l in the log2 domain, P = exp2(s - m) split as
//         a bf16 pair P_hi + P_lo (R13) written to shared memory in the 128-byte
//         swizzled K-major layout the tensor core reads
//   MMA2  O_blk = P_hi V + P_lo V  (M = 128, N = HD head dims, K = BN keys) -> TMEM,
//         V given transposed (V^T[d][key], from a transpose kernel) so both
//         operands are K-major
//   softmax warps: O = O * exp2(m_prev - m) + O_blk in registers.
// S and O_blk are double-buffered in TMEM so MMA1 of the next block overlaps
// the softmax of this one.  The row normaliser is written as lse2 = m +
// log2(l) for the column-mass pass.
//
// Roles (320 threads): warp 0 TMA producer (Q once; K and V^T tiles of each
// key block, two stages), warp 1 MMA issuer, warps 2..9 softmax/epilogue
// (warp w reads TMEM lanes 32*(w%4)..+32, keys and output dims of half
// (w-2)/4; the halves exchange row maxima and sums through shared memory).  Every wait is bounded; after a
// timeout the roles skip their remaining waits, drain their copies, free TMEM
// and return with the status word set.
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr int AT_BM = 128;  // queries per CTA
constexpr int AT_THREADS = 320;
constexpr int AT_SOFT_WARPS = 8;
constexpr int AT_STAGES = 3;  // K/V^T stages: V stays until MMA2, after the softmax
constexpr uint32_t AT_TMEM_COLS = 512;  // S[2] (2 x BN) + O[2] (2 x HD), rounded to a power of two

// Tile geometry per head size.  Operands are stored as 64-element-wide
// (128-byte) swizzled chunks: Q [128 q x HD] and K [BN x HD] as HD/64 chunks
// over the head dims, V^T [HD x BN] and P [128 q x BN] as BN/64 chunks over
// the keys.
template <int HD>
struct AtCfg {
  static constexpr int BN = HD == 64 ? 128 : 64;  // keys per block
  static constexpr int Q_BYTES = AT_BM * HD * 2;
  static constexpr int K_BYTES = BN * HD * 2;
  static constexpr int V_BYTES = HD * BN * 2;
  static constexpr int P_BYTES = AT_BM * BN * 2;
  // Q[2] | K[STAGES] | V^T[STAGES] | P_hi | P_lo | barriers | row-max exchange
  // [2][2][128] | row-sum exchange [2][128]; +1 KB to align to the swizzle atom
  static constexpr size_t SMEM = 2 * Q_BYTES + AT_STAGES * (K_BYTES + V_BYTES) + 2 * P_BYTES + 256 +
                                 6 * AT_BM * 4 + 1024;
  static constexpr int O_COL = 2 * BN;  // TMEM column of O[0]
};
static_assert(AtCfg<64>::SMEM <= 227 * 1024 && AtCfg<128>::SMEM <= 227 * 1024, "shared memory");
static_assert(2 * AtCfg<64>::BN + 2 * 64 <= 512 && 2 * AtCfg<128>::BN + 2 * 128 <= 512, "TMEM columns");

struct AtArgs {
  float* lse2;  // [B, Hq, N]
  bf16* out;    // [B*N, Hq*HD]
  int B, N, Hq, Hkv, n_qb, causal;  // grid: persistent, one CTA per SM
  float scale_log2;
  int* status;
};

// 2^x on the special-function unit (flush-to-zero: P entries below 2^-126 are
// zero next to the row's maximum entry of 1).
__device__ __forceinline__ float ex2_fast(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t swz128(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// Work item t (longest query blocks first): query block, head, sequence.
struct AtItem {
  int qb, h, b, n_kb;
};
template <int BN>
__device__ __forceinline__ AtItem at_item(int t, const AtArgs& a) {
  AtItem it;
  const int per_qb = a.Hq * a.B;
  it.qb = a.n_qb - 1 - t / per_qb;
  const int r = t % per_qb;
  it.h = r % a.Hq;
  it.b = r / a.Hq;
  // causal: the key blocks up to the last query of the block (or the sequence)
  const int keys = a.causal ? min(a.N, (it.qb + 1) * AT_BM) : a.N;
  it.n_kb = (keys + BN - 1) / BN;
  return it;
}

template <int HD>
__global__ void __launch_bounds__(AT_THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_vt, const AtArgs a) {
  using C = AtCfg<HD>;
  constexpr int AT_BN = C::BN, AT_HD = HD;
  constexpr int AT_Q_BYTES = C::Q_BYTES, AT_K_BYTES = C::K_BYTES, AT_V_BYTES = C::V_BYTES,
                AT_P_BYTES = C::P_BYTES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;                                // [2]
  uint8_t* sK = sQ + 2 * AT_Q_BYTES;                 // [AT_STAGES]
  uint8_t* sV = sK + AT_STAGES * AT_K_BYTES;         // [AT_STAGES]
  uint8_t* sPh = sV + AT_STAGES * AT_V_BYTES;
  uint8_t* sPl = sPh + AT_P_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sPl + AT_P_BYTES);
  uint64_t* q_full = bars;            // [2]
  uint64_t* q_empty = bars + 2;       // [2]
  uint64_t* kv_full = bars + 4;       // [AT_STAGES]
  uint64_t* kv_empty = bars + 7;      // [AT_STAGES]
  uint64_t* s_full = bars + 10;       // [2]
  uint64_t* s_empty = bars + 12;      // [2]
  uint64_t* p_full = bars + 14;       // [1]
  uint64_t* p_empty = bars + 15;      // [1]
  uint64_t* o_full = bars + 16;       // [2]
  uint64_t* o_empty = bars + 18;      // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 20);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* s_rowmax = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int total = a.n_qb * a.Hq * a.B;
  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int i = 0; i < AT_STAGES; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&q_full[i], 1);
      mbar_init(&q_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], AT_SOFT_WARPS);
      mbar_init(&o_full[i], 1);
      mbar_init(&o_empty[i], AT_SOFT_WARPS);
    }
    mbar_init(p_full, AT_SOFT_WARPS);
    mbar_init(p_empty, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tm_q);
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_vt);
  }
  if (warp == 1) tmem_alloc(tmem_slot, AT_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();

  // J counts the key blocks this CTA has streamed over all its items; the K/V
  // stages, S and O buffers alternate with J, the Q buffers with the item count.
  if (warp == 0) {
    if (lane == 0) {
      bool ok = true;
      uint32_t J = 0, items = 0, q_issued = 0;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++items) {
        const AtItem it = at_item<AT_BN>(t, a);
        const int g = it.h / (a.Hq / a.Hkv);
        const int row0 = it.b * a.N;
        const int qs = items & 1;
        if (!mbar_wait_ab(&q_empty[qs], ((items >> 1) & 1) ^ 1, a.status, abort_flag)) {
          ok = false;
          break;
        }
        ++q_issued;
        mbar_arrive_expect_tx(&q_full[qs], AT_Q_BYTES);
        for (int c = 0; c < AT_HD / 64; ++c)
          tma_load_2d(sQ + qs * AT_Q_BYTES + c * (AT_BM * 128), &tm_q, it.h * AT_HD + c * 64,
                      row0 + it.qb * AT_BM, &q_full[qs]);
        for (int j = 0; j < it.n_kb; ++j, ++J) {
          const int st = J % AT_STAGES;
          if (!mbar_wait_ab(&kv_empty[st], ((J / AT_STAGES) & 1) ^ 1, a.status, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&kv_full[st], AT_K_BYTES + AT_V_BYTES);
          for (int c = 0; c < AT_HD / 64; ++c)
            tma_load_2d(sK + st * AT_K_BYTES + c * (AT_BN * 128), &tm_k, (a.Hq + g) * AT_HD + c * 64,
                        row0 + j * AT_BN, &kv_full[st]);
          for (int c = 0; c < AT_BN / 64; ++c)
            tma_load_2d(sV + st * AT_V_BYTES + c * (AT_HD * 128), &tm_vt, j * AT_BN + c * 64,
                        (it.b * a.Hkv + g) * AT_HD, &kv_full[st]);
        }
      }
      if (!ok) {  // let the copies already issued land before the CTA's memory goes away
        for (uint32_t k = J; k > 0 && k + AT_STAGES > J; --k)
          mbar_wait(&kv_full[(k - 1) % AT_STAGES], ((k - 1) / AT_STAGES) & 1, nullptr);
        for (uint32_t k = q_issued; k > 0 && k + 2 > q_issued; --k)
          mbar_wait(&q_full[(k - 1) & 1], ((k - 1) >> 1) & 1, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(AT_BM, AT_BN);
      constexpr uint32_t idesc_o = idesc_bf16_f32(AT_BM, AT_HD);
      bool ok = true;
      auto mma2 = [&](uint32_t J) -> bool {  // O[J&1] = P_hi V_J + P_lo V_J
        const int ob = J & 1;
        if (!mbar_wait_ab(p_full, J & 1, a.status, abort_flag)) return false;
        if (!mbar_wait_ab(&o_empty[ob], ((J >> 1) & 1) ^ 1, a.status, abort_flag)) return false;
        tc_fence_after();
        const uint32_t v_base = smem_u32(sV + (J % AT_STAGES) * AT_V_BYTES);
        const uint32_t d_tmem = tmem + C::O_COL + ob * AT_HD;
#pragma unroll
        for (int part = 0; part < 2; ++part) {
          const uint32_t p_base = smem_u32(part ? sPl : sPh);
#pragma unroll
          for (int kk = 0; kk < AT_BN / 16; ++kk) {  // 64-key chunk kk/4 of P and of V^T
            const uint32_t pa = p_base + (kk / 4) * (AT_BM * 128) + (kk % 4) * 32;
            const uint32_t va = v_base + (kk / 4) * (AT_HD * 128) + (kk % 4) * 32;
            tc_mma_bf16(d_tmem, sdesc_sw128(pa), sdesc_sw128(va), idesc_o, (part | kk) ? 1u : 0u);
          }
        }
        tc_commit(&o_full[ob]);
        tc_commit(p_empty);
        tc_commit(&kv_empty[J % AT_STAGES]);
        return true;
      };
      uint32_t J = 0, items = 0;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++items) {
        const AtItem it = at_item<AT_BN>(t, a);
        const int qs = items & 1;
        if (!mbar_wait_ab(&q_full[qs], (items >> 1) & 1, a.status, abort_flag)) {
          ok = false;
          break;
        }
        const uint32_t q_base = smem_u32(sQ + qs * AT_Q_BYTES);
        for (int j = 0; j < it.n_kb; ++j, ++J) {
          const int kst = J % AT_STAGES, sb = J & 1;
          if (!mbar_wait_ab(&kv_full[kst], (J / AT_STAGES) & 1, a.status, abort_flag) ||
              !mbar_wait_ab(&s_empty[sb], ((J >> 1) & 1) ^ 1, a.status, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t k_base = smem_u32(sK + kst * AT_K_BYTES);
          const uint32_t d_tmem = tmem + sb * AT_BN;
#pragma unroll
          for (int kk = 0; kk < AT_HD / 16; ++kk)  // 64-dim chunk kk/4 of Q and of K
            tc_mma_bf16(d_tmem, sdesc_sw128(q_base + (kk / 4) * (AT_BM * 128) + (kk % 4) * 32),
                        sdesc_sw128(k_base + (kk / 4) * (AT_BN * 128) + (kk % 4) * 32), idesc_s,
                        kk > 0 ? 1u : 0u);
          tc_commit(&s_full[sb]);
          if (j + 1 == it.n_kb) tc_commit(&q_empty[qs]);  // this item's Q is read for the last time
          if (J > 0 && !mma2(J - 1)) {
            ok = false;
            break;
          }
        }
      }
      if (ok && J > 0) mma2(J - 1);
    }
    __syncwarp();
  } else {
    // softmax and output: thread = query row of the item; the two warps on a
    // TMEM lane quadrant split the row (keys half*64.., output dims half*32..)
    const int ew = warp - 2;
    const int quad = warp & 3, half = ew / 4;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    constexpr int KH = AT_BN / 2, OH = AT_HD / 2;
    float corr_ring[2] = {1.f, 1.f};
    bool ok = true;
    auto arrive = [&](uint64_t* bar) {
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
    };
    uint32_t J = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      const AtItem it = at_item<AT_BN>(t, a);
      const int q0 = it.qb * AT_BM, q = q0 + row;
      float m = -INFINITY, l = 0.f;
      float o[OH];
#pragma unroll
      for (int e = 0; e < OH; ++e) o[e] = 0.f;
      auto merge = [&](uint32_t Jm) {  // O = O * corr + O_blk(Jm), this warp's 32 dims
        const int ob = Jm & 1;
        ok = ok && __all_sync(0xffffffffu, mbar_wait_ab(&o_full[ob], (Jm >> 1) & 1, a.status, abort_flag));
        tc_fence_after();
        if (ok) {
          const float cj = corr_ring[Jm & 1];
          const uint32_t oaddr = tmem + lane_off + C::O_COL + ob * AT_HD + half * OH;
#pragma unroll
          for (int c = 0; c < OH; c += 32) {
            uint32_t r[32];
            __syncwarp();
            tmem_ld16(oaddr + c, *reinterpret_cast<uint32_t(*)[16]>(r));
            tmem_ld16(oaddr + c + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[c + e] = fmaf(o[c + e], cj, __uint_as_float(r[e]));
          }
        }
        tc_fence_before();
        arrive(&o_empty[ob]);
      };
      for (int j = 0; j < it.n_kb; ++j, ++J) {
        const int st = J & 1;
        ok = ok && __all_sync(0xffffffffu, mbar_wait_ab(&s_full[st], (J >> 1) & 1, a.status, abort_flag));
        tc_fence_after();
        // this warp's 64 columns of the S row, raw scores kept in registers;
        // masked entries become -inf (only the diagonal and the last block mask)
        const int k0 = j * AT_BN + half * KH;
        const bool diag = a.causal && j * AT_BN + AT_BN > q0;  // causal mask inside this block
        const bool tail = k0 + KH > a.N;                        // keys past the sequence
        uint32_t r[KH];
        float mx = -INFINITY;
        if (ok) {
          const uint32_t s_addr = tmem + lane_off + st * AT_BN + half * KH;
          __syncwarp();
#pragma unroll
          for (int c = 0; c < KH; c += 16) tmem_ld16(s_addr + c, *reinterpret_cast<uint32_t(*)[16]>(r + c));
          tmem_ld_wait();
          if (diag || tail) {  // keys k0 + e with e >= lim are hidden
            int lim = KH;
            if (diag) lim = min(lim, q - k0 + 1);
            if (tail) lim = min(lim, a.N - k0);
#pragma unroll
            for (int e = 0; e < KH; ++e)
              if (e >= lim) r[e] = __float_as_uint(-INFINITY);
          }
#pragma unroll
          for (int e = 0; e < KH; ++e) mx = fmaxf(mx, __uint_as_float(r[e]));
        }
        tc_fence_before();
        arrive(&s_empty[st]);  // S is in registers now
        // the row maximum over both halves (exchange buffer alternates with J);
        // the scale is positive, so max(s * c) = c * max(s)
        s_rowmax[(J & 1) * 2 * AT_BM + half * AT_BM + row] = mx;
        asm volatile("bar.sync 1, %0;" ::"n"(AT_SOFT_WARPS * 32) : "memory");
        mx = fmaxf(mx, s_rowmax[(J & 1) * 2 * AT_BM + (half ^ 1) * AT_BM + row]);
        const float m_new = fmaxf(m, mx == -INFINITY ? -INFINITY : mx * a.scale_log2);
        const float base = m_new == -INFINITY ? 0.f : m_new;
        corr_ring[J & 1] = exp2f(m - base);
        l *= corr_ring[J & 1];
        m = m_new;
        // P_J: wait until MMA2 of block J-1 has read the P buffer
        ok = ok && __all_sync(0xffffffffu, mbar_wait_ab(p_empty, (J & 1) ^ 1, a.status, abort_flag));
        if (ok) {
#pragma unroll
          for (int c = 0; c < KH / 8; ++c) {  // 16-byte chunk c: keys half*KH + 8c .. +7
            uint32_t hi[4], lo[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float p0 = ex2_fast(fmaf(__uint_as_float(r[8 * c + 2 * e]), a.scale_log2, -base));
              const float p1 = ex2_fast(fmaf(__uint_as_float(r[8 * c + 2 * e + 1]), a.scale_log2, -base));
              l += p0 + p1;
              hi[e] = pack_bf16x2(p0, p1);
              lo[e] = pack_bf16x2(p0 - bf16lo(hi[e]), p1 - bf16hi(hi[e]));
            }
            const int key = half * KH + 8 * c;  // in 64-key chunk key/64, 16-byte unit (key%64)/8
            const uint32_t off = (key / 64) * (AT_BM * 128) + swz128(row, (key % 64) / 8);
            *reinterpret_cast<uint4*>(sPh + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
            *reinterpret_cast<uint4*>(sPl + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
          }
        }
        fence_proxy_async_smem();  // the tensor core reads P through the async proxy
        arrive(p_full);
        if (j > 0) merge(J - 1);
      }
      merge(J - 1);  // this item's last block
      // total normaliser of the row = the two halves' sums (own exchange buffer)
      s_rowmax[4 * AT_BM + half * AT_BM + row] = l;
      asm volatile("bar.sync 1, %0;" ::"n"(AT_SOFT_WARPS * 32) : "memory");
      const float l_all = l + s_rowmax[4 * AT_BM + (half ^ 1) * AT_BM + row];
      asm volatile("bar.sync 1, %0;" ::"n"(AT_SOFT_WARPS * 32) : "memory");  // buffer reusable
      if (ok && q < a.N) {
        const float inv = l_all > 0.f ? 1.f / l_all : 0.f;
        bf16* orow = a.out + (static_cast<size_t>(it.b) * a.N + q) * (static_cast<size_t>(a.Hq) * AT_HD) +
                     it.h * AT_HD + half * OH;
#pragma unroll
        for (int c = 0; c < OH; c += 8) {
          uint4 v;
          v.x = pack_bf16x2(o[c] * inv, o[c + 1] * inv);
          v.y = pack_bf16x2(o[c + 2] * inv, o[c + 3] * inv);
          v.z = pack_bf16x2(o[c + 4] * inv, o[c + 5] * inv);
          v.w = pack_bf16x2(o[c + 6] * inv, o[c + 7] * inv);
          *reinterpret_cast<uint4*>(orow + c) = v;
        }
        if (half == 0) a.lse2[(static_cast<size_t>(it.b) * a.Hq + it.h) * a.N + q] = m + log2f(l_all);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, AT_TMEM_COLS);
  }
}

// vt[(b*Hkv + g)*HD + d][j] = v of key j, group g, dim d (keys past N: zero up to ldt).
template <int AT_HD>
__global__ void v_transpose_kernel(const bf16* __restrict__ qkv, int B, int N, int Hq, int Hkv,
                                   int ldt, bf16* __restrict__ vt) {
  pdl_trigger();
  pdl_wait();
  __shared__ bf16 tile[32][33];
  const int bg = blockIdx.z, b = bg / Hkv, g = bg % Hkv;
  const int j0 = blockIdx.x * 32, d0 = blockIdx.y * 32;
  const size_t ld = static_cast<size_t>(Hq + 2 * Hkv) * AT_HD;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8
  for (int r = ty; r < 32; r += 8) {
    const int j = j0 + r;
    tile[r][tx] = j < N ? qkv[(static_cast<size_t>(b) * N + j) * ld + static_cast<size_t>(Hq + Hkv + g) * AT_HD + d0 + tx]
                        : __float2bfloat16_rn(0.f);
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    const int j = j0 + tx;
    if (j < ldt) vt[(static_cast<size_t>(bg) * AT_HD + d0 + r) * ldt + j] = tile[tx][r];
  }
}

// SMs of the current device (kept per device).
int attn_sms() {
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

bool encode(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t ld_elems,
            uint32_t box_inner, uint32_t box_rows) {
  EncodeTiledFn enc = get_encode_tiled();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {ld_elems * 2};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

size_t attention_tc_vt_elems(int B, int N, int Hkv, int hd) {
  return static_cast<size_t>(B) * Hkv * hd * ((N + 7) & ~7);
}

bool attention_tc_supported(int dtype, int hd, const int* cu, const uint8_t* key_alive, int* status,
                            void* vt) {
  return dtype == ZSAA_BF16 && (hd == 64 || hd == 128) && cu == nullptr && key_alive == nullptr &&
         status != nullptr && vt != nullptr;
}

// Measured on the 1B heads (B = 8): the tcgen05 kernel and its V transpose beat
// the mma.sync kernel from about two 128-row query blocks on; below, the
// extra launch and 128-row tiles on short sequences cost more than they save.
bool attention_tc_preferred(int N) { return N >= kAttentionTcMinN; }

namespace {

template <int HD>
cudaError_t run_attention_tc(const void* qkv, void* vt, int B, int N, int Hq, int Hkv, void* out,
                             float* lse, int causal, int* status, cudaStream_t s) {
  using C = AtCfg<HD>;
  const int ldt = (N + 7) & ~7;
  const int ld = (Hq + 2 * Hkv) * HD;
  {
    dim3 grid((ldt + 31) / 32, HD / 32, B * Hkv);
    ZSAA_LAUNCH(v_transpose_kernel<HD>, grid, dim3(256), 0, s, static_cast<const bf16*>(qkv), B, N, Hq, Hkv,
                ldt, static_cast<bf16*>(vt));
  }
  CUtensorMap tm_q, tm_k, tm_vt;
  if (!encode(&tm_q, qkv, static_cast<uint64_t>(ld), static_cast<uint64_t>(B) * N, ld, 64, AT_BM))
    return cudaErrorInvalidValue;
  if (!encode(&tm_k, qkv, static_cast<uint64_t>(ld), static_cast<uint64_t>(B) * N, ld, 64, C::BN))
    return cudaErrorInvalidValue;
  if (!encode(&tm_vt, vt, static_cast<uint64_t>(ldt), static_cast<uint64_t>(B) * Hkv * HD, ldt, 64, HD))
    return cudaErrorInvalidValue;
  static OncePerDevice once;
  const cudaError_t attr_err = set_smem_limit_once(once, attn_tc_kernel<HD>, static_cast<int>(C::SMEM));
  if (attr_err != cudaSuccess) return attr_err;
  AtArgs a;
  a.lse2 = lse;
  a.out = static_cast<bf16*>(out);
  a.B = B;
  a.N = N;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.n_qb = (N + AT_BM - 1) / AT_BM;
  a.causal = causal;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
  a.status = status;
  const int total = a.n_qb * Hq * B;
  const int grid = total < attn_sms() ? total : attn_sms();
  ZSAA_LAUNCH(attn_tc_kernel<HD>, dim3(grid), dim3(AT_THREADS), C::SMEM, s, tm_q, tm_k, tm_vt, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attention_tc(const void* qkv, void* vt, int B, int N, int Hq, int Hkv, int hd,
                                void* out, float* lse, int causal, int* status, cudaStream_t s) {
  if (hd == 64) return run_attention_tc<64>(qkv, vt, B, N, Hq, Hkv, out, lse, causal, status, s);
  if (hd == 128) return run_attention_tc<128>(qkv, vt, B, N, Hq, Hkv, out, lse, causal, status, s);
  return cudaErrorInvalidValue;
}

}  // namespace zsaa
