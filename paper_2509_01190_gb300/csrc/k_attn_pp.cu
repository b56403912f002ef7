// Causal (or bidirectional) grouped-query attention, Eq. 1, on the sm_103a
// tensor cores: two query tiles per CTA whose softmaxes take turns, so each
// tile's exponentials run while the tensor core works on the other tile.
//
// A work item is (sequence b, KV group g, pair of query heads h0 and h0+1 of
// that group, block of 128 queries).  Both heads read the same keys and
// values, so each K/V block is loaded once for the two tiles.  Per key block
// j of 128 keys (causal: up to the diagonal):
//   S_x = Q_x K_j^T                      (tcgen05, M = 128, N = 128, K = hd)
//   softmax warps of tile x (one query row per thread, TMEM lane = row):
//     pass 1: the block's row maximum (masked keys excluded), log2 domain;
//       the running maximum m moves only when the block's exceeds it by more
//       than 2^8 (until then P entries may reach 256, exact in fp32 and in the
//       bf16 pair), and then O is rescaled in TMEM by 2^(m_old - m_new);
//     pass 2: P = 2^(s*scale - m) as a bf16 pair P_hi + P_lo (P_lo is the
//       rounding remainder, so P is carried to ~16 bits), written back over
//       the S columns it came from, and the running row sum l.
//   O_x += P_hi V_j + P_lo V_j           (A = P from TMEM, B = V straight from
//                                         the packed qkv rows, MN-major)
// O stays in TMEM across the key blocks; the epilogue divides by l, rounds to
// bf16 and writes the row normaliser lse2 = m + log2(l).
//
// Tensor-core order (one issuing thread; tcgen05.mma executes in issue order):
//   S_A(0) S_B(0) | PV_A(0) S_A(1) PV_B(0) S_B(1) | PV_A(1) S_A(2) PV_B(1) ...
// so tile A's softmax of block j+1 runs under PV_B(j) and S_B(j+1), and tile
// B's under PV_A(j+1) and S_A(j+2).
//
// Roles (384 threads): warp 0 TMA producer (both Q tiles per item; K and V of
// every key block through a ring), warp 1 MMA issuer, warps 4-7 tile A's
// softmax and epilogue, warps 8-11 tile B's (warp w reads TMEM lanes
// 32*(w%4)..+31).  TMEM: S_A | O_A | S_B | O_B, 128 columns each.  Every wait
// is bounded; after a timeout every role skips its remaining work, copies in
// flight are drained, and TMEM is freed.
#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr int PP_BM = 128;  // queries per tile
constexpr int PP_BN = 128;  // keys per block
constexpr int PP_THREADS = 384;
constexpr uint32_t PP_TMEM_COLS = 512;
constexpr float PP_RESCALE_LOG2 = 8.0f;  // lazy rescale threshold (factor 256)

template <int HD>
struct PpCfg {
  static constexpr int CH = HD / 64;                 // 64-dim (128-byte) chunks
  static constexpr int TILE = PP_BM * HD * 2;        // one Q tile, K block or V block
  static constexpr int STAGES = HD == 128 ? 2 : 4;   // K/V ring
  static constexpr size_t SMEM = 2 * static_cast<size_t>(TILE) + 2 * STAGES * static_cast<size_t>(TILE) + 256 + 1024;
};
static_assert(PpCfg<64>::SMEM <= 227 * 1024 && PpCfg<128>::SMEM <= 227 * 1024, "shared memory");

__host__ __device__ constexpr uint32_t s_col(int x) { return 256u * x; }
__host__ __device__ constexpr uint32_t o_col(int x) { return 256u * x + 128u; }

struct PpArgs {
  float* lse2;  // [B, Hq, N], log2 domain
  bf16* out;    // [B*N, Hq*hd]
  int B, N, Hq, Hkv, pairs, n_qb, causal;
  float scale_log2;
  int* status;
};

struct PpItem {
  int qb, b, g, h0, n_kb;
};

// The r-th work item of this CTA: items are numbered longest query blocks
// first and dealt to the CTAs in a snake order (0..G-1, then G-1..0, ...), so
// the causal triangle's long and short items even out across CTAs.  Returns
// an index >= total once the CTA has none left (the sequence only grows).
__device__ __forceinline__ int pp_item_index(int r) {
  const int G = gridDim.x, i = blockIdx.x;
  return r * G + ((r & 1) ? G - 1 - i : i);
}

// Work item t, longest query blocks first.
__device__ __forceinline__ PpItem pp_item(int t, const PpArgs& a) {
  PpItem it;
  const int per_qb = a.B * a.Hkv * a.pairs;
  it.qb = a.n_qb - 1 - t / per_qb;
  int r = t % per_qb;
  const int hp = r % a.pairs;
  r /= a.pairs;
  it.g = r % a.Hkv;
  it.b = r / a.Hkv;
  it.h0 = it.g * (a.Hq / a.Hkv) + 2 * hp;
  const int keys = a.causal ? min(a.N, (it.qb + 1) * PP_BM) : a.N;
  it.n_kb = (keys + PP_BN - 1) / PP_BN;
  return it;
}

__device__ __forceinline__ float ex2_fast(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Shared-memory descriptor of an MN-major operand with the 128-byte swizzle:
// rows of 64 bf16 along N (128 B) for consecutive K, 8-row atoms 1024 B apart
// along K (stride byte offset), 64-element N chunks `chunk_bytes` apart
// (leading byte offset).
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t saddr, uint32_t chunk_bytes) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((chunk_bytes >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// D[tmem] (+)= A[tmem] * B[smem]: A (M x K) read from tensor memory, lane =
// row, two bf16 per 32-bit column in K order (lower K in the low half).
__device__ __forceinline__ void tc_mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                               uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Warp-collective: lane i reads / writes TMEM lane (base + i), 32 consecutive columns.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}


__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  tmem_st16(taddr, *reinterpret_cast<const uint32_t(*)[16]>(r));
  tmem_st16(taddr + 16, *reinterpret_cast<const uint32_t(*)[16]>(r + 16));
}


template <int HD>
__global__ void __launch_bounds__(PP_THREADS, 1)
    attn_pp_kernel(const __grid_constant__ CUtensorMap tm, const PpArgs a) {
  using C = PpCfg<HD>;
  constexpr int CH = C::CH, TILE = C::TILE, ST = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;                   // [2 tiles]
  uint8_t* sK = sQ + 2 * TILE;          // [ST]
  uint8_t* sV = sK + ST * TILE;         // [ST]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + ST * TILE);
  uint64_t* q_full = bars;              // [1]
  uint64_t* q_empty = bars + 1;         // [1]
  uint64_t* s_full = bars + 2;          // [2] per tile
  uint64_t* p_full = bars + 4;          // [2]
  uint64_t* o_full = bars + 6;          // [2]
  uint64_t* o_empty = bars + 8;         // [2]
  uint64_t* mma_done = bars + 10;       // [1]
  uint64_t* kv_full = bars + 11;        // [ST]
  uint64_t* kv_empty = bars + 11 + ST;  // [ST]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11 + 2 * ST);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int total = a.n_qb * a.B * a.Hkv * a.pairs;
  pdl_trigger();
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int x = 0; x < 2; ++x) {
      mbar_init(&s_full[x], 1);
      mbar_init(&p_full[x], 4);
      mbar_init(&o_full[x], 1);
      mbar_init(&o_empty[x], 4);
    }
    mbar_init(mma_done, 1);
    for (int i = 0; i < ST; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) prefetch_tmap(&tm);
  if (warp == 1) tmem_alloc(tmem_slot, PP_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      bool ok = true;
      uint32_t J = 0, items = 0, q_issued = 0;
      for (int t = pp_item_index(0); t < total && ok; t = pp_item_index(++items)) {
        const PpItem it = pp_item(t, a);
        const int row0 = it.b * a.N;
        if (!mbar_wait_ab(q_empty, (items & 1) ^ 1, a.status, abort_flag)) {
          ok = false;
          break;
        }
        ++q_issued;
        mbar_arrive_expect_tx(q_full, 2 * TILE);
        for (int x = 0; x < 2; ++x)
          for (int c = 0; c < CH; ++c)
            tma_load_2d(sQ + x * TILE + c * (PP_BM * 128), &tm, (it.h0 + x) * HD + c * 64,
                        row0 + it.qb * PP_BM, q_full);
        for (int j = 0; j < it.n_kb; ++j, ++J) {
          const int st = J % ST;
          if (!mbar_wait_ab(&kv_empty[st], ((J / ST) & 1) ^ 1, a.status, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&kv_full[st], 2 * TILE);
          for (int c = 0; c < CH; ++c) {
            tma_load_2d(sK + st * TILE + c * (PP_BN * 128), &tm, (a.Hq + it.g) * HD + c * 64,
                        row0 + j * PP_BN, &kv_full[st]);
            tma_load_2d(sV + st * TILE + c * (PP_BN * 128), &tm, (a.Hq + a.Hkv + it.g) * HD + c * 64,
                        row0 + j * PP_BN, &kv_full[st]);
          }
        }
      }
      if (!ok) {  // let the copies already issued land before the CTA's memory goes away
        for (uint32_t k = J; k > 0 && k + ST > J; --k)
          mbar_wait(&kv_full[(k - 1) % ST], ((k - 1) / ST) & 1, nullptr);
        if (q_issued > 0) mbar_wait(q_full, (q_issued - 1) & 1, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(PP_BM, PP_BN);
      constexpr uint32_t idesc_o = idesc_bf16_f32(PP_BM, HD) | (1u << 16);  // B (V) MN-major
      // V's 64-dim chunks are PP_BN * 128 bytes apart; with one chunk (hd 64)
      // the stride is never used and is set to the 8-row atom stride, so the
      // descriptor addresses only the 16 keys of each MMA either way.
      constexpr uint32_t kVChunkStride = CH > 1 ? PP_BN * 128 : 1024;
      bool ok = true;
      uint32_t J = 0, items = 0;
      auto issue_s = [&](int x, int st) {  // S_x = Q_x K^T
        const uint32_t qa = smem_u32(sQ + x * TILE), ka = smem_u32(sK + st * TILE);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          tc_mma_bf16(tmem + s_col(x), sdesc_sw128(qa + (kk / 4) * (PP_BM * 128) + (kk % 4) * 32),
                      sdesc_sw128(ka + (kk / 4) * (PP_BN * 128) + (kk % 4) * 32), idesc_s, kk > 0 ? 1u : 0u);
        tc_commit(&s_full[x]);
      };
      auto issue_pv = [&](int x, int st, bool first) {  // O_x (+)= P_hi V + P_lo V
        const uint32_t va = smem_u32(sV + st * TILE);
#pragma unroll
        for (int part = 0; part < 2; ++part)
#pragma unroll
          for (int kk = 0; kk < PP_BN / 16; ++kk)
            tc_mma_bf16_ts(tmem + o_col(x), tmem + s_col(x) + 32 * (kk / 2) + 16 * part + 8 * (kk % 2),
                           sdesc_sw128_mn(va + kk * 16 * 128, kVChunkStride), idesc_o,
                           (first && part == 0 && kk == 0) ? 0u : 1u);
      };
      for (int t = pp_item_index(0); t < total && ok; t = pp_item_index(++items)) {
        const PpItem it = pp_item(t, a);
        if (!mbar_wait_ab(q_full, items & 1, a.status, abort_flag)) {
          ok = false;
          break;
        }
        for (int j = 0; j < it.n_kb && ok; ++j) {
          const uint32_t Jj = J + j;
          const int st = Jj % ST;
          if (j == 0) {
            if (!mbar_wait_ab(&kv_full[st], (Jj / ST) & 1, a.status, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_s(0, st);
            issue_s(1, st);
            if (it.n_kb == 1) tc_commit(q_empty);
          }
          const bool more = j + 1 < it.n_kb;
          const int st1 = (Jj + 1) % ST;
          for (int x = 0; x < 2 && ok; ++x) {
            // the epilogue of the previous item has read O_x out
            if (j == 0 && items > 0 && !mbar_wait_ab(&o_empty[x], (items - 1) & 1, a.status, abort_flag)) {
              ok = false;
              break;
            }
            if (!mbar_wait_ab(&p_full[x], Jj & 1, a.status, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_pv(x, st, j == 0);
            if (x == 1) tc_commit(&kv_empty[st]);  // K_j and V_j read for the last time
            if (more) {
              if (x == 0) {
                if (!mbar_wait_ab(&kv_full[st1], ((Jj + 1) / ST) & 1, a.status, abort_flag)) {
                  ok = false;
                  break;
                }
                tc_fence_after();
              }
              issue_s(x, st1);
              if (x == 1 && j + 2 == it.n_kb) tc_commit(q_empty);  // Q read for the last time
            } else {
              tc_commit(&o_full[x]);
            }
          }
        }
        J += it.n_kb;
      }
      // every MMA issued has finished before the CTA frees TMEM
      tc_commit(mma_done);
      mbar_wait(mma_done, 0, a.status);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---------------------------------------------------------------- softmax + epilogue
    const int x = (warp - 4) / 4;  // tile
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t s_addr = tmem + lane_off + s_col(x);
    const uint32_t o_addr = tmem + lane_off + o_col(x);
    bool ok = true;
    uint32_t J = 0, items = 0;
    auto arrive = [&](uint64_t* bar) {
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
    };
    for (int t = pp_item_index(0); t < total; t = pp_item_index(++items)) {
      const PpItem it = pp_item(t, a);
      const int q = it.qb * PP_BM + row;
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < it.n_kb; ++j) {
        const uint32_t Jj = J + j;
        ok = ok && __all_sync(0xffffffffu, mbar_wait_ab(&s_full[x], Jj & 1, a.status, abort_flag));
        tc_fence_after();
        // keys k0 + e with e >= lim are hidden (causal diagonal, sequence end)
        const int k0 = j * PP_BN;
        int lim = min(PP_BN, a.N - k0);
        if (a.causal) lim = min(lim, q - k0 + 1);
        if (ok) {
          // masking (causal diagonal or sequence end) only where some lane of
          // the warp needs it, so full blocks take the branch-free path
          const bool masked = __any_sync(0xffffffffu, lim < PP_BN);
          // pass 1: the block's row maximum, 64 columns per TMEM round trip
          float mx = -INFINITY;
#pragma unroll 1
          for (int c = 0; c < PP_BN / 32; c += 2) {
            uint32_t r[64];
            tmem_ld32(s_addr + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(r));
            tmem_ld32(s_addr + 32 * c + 32, *reinterpret_cast<uint32_t(*)[32]>(r + 32));
            tmem_ld_wait();
            if (!masked) {
#pragma unroll
              for (int e = 0; e < 64; ++e) mx = fmaxf(mx, __uint_as_float(r[e]));
            } else {
#pragma unroll
              for (int e = 0; e < 64; ++e)
                if (32 * c + e < lim) mx = fmaxf(mx, __uint_as_float(r[e]));
            }
          }
          const float mb = mx == -INFINITY ? -INFINITY : mx * a.scale_log2;
          const bool need = mb > m + PP_RESCALE_LOG2;
          if (__any_sync(0xffffffffu, need)) {
            const float mn = need ? mb : m;
            const float f = need ? (m == -INFINITY ? 0.f : exp2f(m - mn)) : 1.f;
            if (j > 0) {  // O holds blocks 0..j-1 (PV_x(j-1) finished before S_x(j) was signalled)
#pragma unroll 1
              for (int c = 0; c < HD / 32; ++c) {
                uint32_t r[32];
                tmem_ld32(o_addr + 32 * c, r);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * f);
                tmem_st32(o_addr + 32 * c, r);
              }
            }
            l *= f;
            m = mn;
          }
          // pass 2: P as a bf16 pair over the S columns just read; the next
          // chunk's load is in flight while this one is converted
          // P = 2^(s*scale - m) split as hi = P rounded to bf16 and lo = P - hi
          // (exact in fp32, then rounded to bf16), so hi + lo carries P to
          // about 17 bits
          const uint64_t scale2 = f2pack(a.scale_log2, a.scale_log2);
          const uint64_t nm2 = f2pack(-m, -m);
          auto emit = [&](const uint32_t (&r)[32], int c) {
            uint32_t hi[16], lo[16];
            uint64_t lsum = f2pack(0.f, 0.f);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              float t0, t1;
              f2unpack(ffma2(f2pack(__uint_as_float(r[2 * e]), __uint_as_float(r[2 * e + 1])), scale2, nm2), t0, t1);
              float p0 = ex2_fast(t0), p1 = ex2_fast(t1);
              if (masked) {
                const int k = 32 * c + 2 * e;
                p0 = k < lim ? p0 : 0.f;
                p1 = k + 1 < lim ? p1 : 0.f;
              }
              const uint64_t pp = f2pack(p0, p1);
              lsum = fadd2(lsum, pp);
              hi[e] = pack_bf16x2(p0, p1);
              float r0, r1;
              f2unpack(fsub2(pp, f2pack(bf16lo(hi[e]), bf16hi(hi[e]))), r0, r1);
              lo[e] = pack_bf16x2(r0, r1);
            }
            float l0, l1;
            f2unpack(lsum, l0, l1);
            l += l0 + l1;
            tmem_st16(s_addr + 32 * c, hi);
            tmem_st16(s_addr + 32 * c + 16, lo);
          };
          uint32_t ra[32], rb[32];
          tmem_ld32(s_addr, ra);
          tmem_ld_wait();
#pragma unroll 1
          for (int c = 0; c < PP_BN / 32; c += 2) {
            tmem_ld32(s_addr + 32 * (c + 1), rb);
            emit(ra, c);
            tmem_ld_wait();
            if (c + 2 < PP_BN / 32) tmem_ld32(s_addr + 32 * (c + 2), ra);
            emit(rb, c + 1);
            tmem_ld_wait();
          }
          tmem_st_wait();
        }
        tc_fence_before();
        arrive(&p_full[x]);
      }
      J += it.n_kb;
      // epilogue: O / l in bf16, and the row normaliser
      ok = ok && __all_sync(0xffffffffu, mbar_wait_ab(&o_full[x], items & 1, a.status, abort_flag));
      tc_fence_after();
      if (ok) {
        const float inv = l > 0.f ? 1.f / l : 0.f;
        const int h = it.h0 + x;
        bf16* orow = a.out + (static_cast<size_t>(it.b) * a.N + q) * (static_cast<size_t>(a.Hq) * HD) + h * HD;
#pragma unroll 1
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(o_addr + 32 * c, r);
          tmem_ld_wait();
          if (q < a.N) {
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              uint4 w;
              w.x = pack_bf16x2(__uint_as_float(r[8 * v + 0]) * inv, __uint_as_float(r[8 * v + 1]) * inv);
              w.y = pack_bf16x2(__uint_as_float(r[8 * v + 2]) * inv, __uint_as_float(r[8 * v + 3]) * inv);
              w.z = pack_bf16x2(__uint_as_float(r[8 * v + 4]) * inv, __uint_as_float(r[8 * v + 5]) * inv);
              w.w = pack_bf16x2(__uint_as_float(r[8 * v + 6]) * inv, __uint_as_float(r[8 * v + 7]) * inv);
              *reinterpret_cast<uint4*>(orow + 32 * c + 8 * v) = w;
            }
          }
        }
        if (q < a.N) a.lse2[(static_cast<size_t>(it.b) * a.Hq + h) * a.N + q] = m + log2f(l);
      }
      tc_fence_before();
      arrive(&o_empty[x]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, PP_TMEM_COLS);
  }
}

int pp_sms() {
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

bool encode_rows(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows) {
  EncodeTiledFn enc = get_encode_tiled();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, 128};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int HD>
cudaError_t run_pp(const void* qkv, int B, int N, int Hq, int Hkv, void* out, float* lse, int causal, int* status,
                   cudaStream_t s) {
  using C = PpCfg<HD>;
  const int ld = (Hq + 2 * Hkv) * HD;
  CUtensorMap tm;
  if (!encode_rows(&tm, qkv, static_cast<uint64_t>(ld), static_cast<uint64_t>(B) * N)) return cudaErrorInvalidValue;
  static OncePerDevice once;
  const cudaError_t attr = set_smem_limit_once(once, attn_pp_kernel<HD>, static_cast<int>(C::SMEM));
  if (attr != cudaSuccess) return attr;
  PpArgs a;
  a.lse2 = lse;
  a.out = static_cast<bf16*>(out);
  a.B = B;
  a.N = N;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.pairs = Hq / Hkv / 2;
  a.n_qb = (N + PP_BM - 1) / PP_BM;
  a.causal = causal;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
  a.status = status;
  const int total = a.n_qb * B * Hkv * a.pairs;
  const int grid = total < pp_sms() ? total : pp_sms();
  ZSAA_LAUNCH(attn_pp_kernel<HD>, dim3(grid), dim3(PP_THREADS), C::SMEM, s, tm, a);
  return cudaGetLastError();
}

}  // namespace

bool attention_pp_supported(int dtype, int hd, int Hq, int Hkv, const int* cu, const uint8_t* key_alive,
                            int* status) {
  return dtype == ZSAA_BF16 && (hd == 64 || hd == 128) && Hkv > 0 && Hq % Hkv == 0 && (Hq / Hkv) % 2 == 0 &&
         cu == nullptr && key_alive == nullptr && status != nullptr;
}

cudaError_t launch_attention_pp(const void* qkv, int B, int N, int Hq, int Hkv, int hd, void* out, float* lse,
                                int causal, int* status, cudaStream_t s) {
  if (B < 1 || N < 1) return cudaSuccess;
  if (hd == 64) return run_pp<64>(qkv, B, N, Hq, Hkv, out, lse, causal, status, s);
  if (hd == 128) return run_pp<128>(qkv, B, N, Hq, Hkv, out, lse, causal, status, s);
  return cudaErrorInvalidValue;
}

}  // namespace zsaa
