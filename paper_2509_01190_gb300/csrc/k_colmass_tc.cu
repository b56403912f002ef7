// Soft-score column mass on the sm_103a tensor cores (Sec. 3.2: soft-score
// times V gives each V row's contribution).
//
// For every sequence b, KV group g, query head h of g and block of 128 keys,
// the CTA computes S^T = K Q^T (M = 128 keys, N = 128 queries, K = hd) with
// tcgen05.mma into TMEM, one query block at a time (only blocks at or after
// the key block when the mask is causal; every block for a bidirectional
// encoder), and its epilogue warps -- one TMEM lane,
// i.e. one key, per thread -- accumulate exp2(s * c - lse2[q]) over the
// queries q >= key of each block.  That is the column sum of the normalised
// soft-score P (the row normalisers lse2 come from the attention kernel).
// Each head writes its own partial, optionally times ||v_key|| of group g (the
// position score of R1 is linear in the column mass; the norms come from the
// QKV projection's epilogue):   parts[hh][b][g][key]
// and the select / reduce kernels sum the Hq/Hkv chunks in a fixed order.
//
// Roles (320 threads): warp 0 TMA producer (K tiles double-buffered, Q tiles
// through a 4-stage ring), warp 1 MMA issuer, warps 2..9 epilogue (warp w
// reads TMEM lanes 32*(w%4)..+32, columns half (w-2)/4 of each 128-query
// block; the halves are added in shared memory at the end of a tile).  Two
// TMEM accumulators let a block's epilogue overlap the next block's MMAs, and
// the next block's query normalisers are fetched with cp.async meanwhile.
// All waits are bounded; epilogue warps never leave the step loop early, so
// their named barriers cannot strand the others.
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr int CM_BM = 128;     // keys per tile (MMA M)
constexpr int CM_BN = 128;     // queries per block (MMA N)
constexpr int CM_STAGES = 4;
constexpr int CM_THREADS = 320;
constexpr int CM_EPI_WARPS = 8;

template <int HD>
struct CmCfg {
  static constexpr int CHUNKS = HD / 64;               // 64-wide swizzled K chunks
  static constexpr int TILE_BYTES = CM_BM * HD * 2;     // K tile or Q tile
  // tiles, then 256 B of barriers and 2 x 128 floats of query normalisers,
  // plus 1 KB to align the tiles to the 128B-swizzle atom
  static constexpr size_t SMEM = static_cast<size_t>(TILE_BYTES) * (2 + CM_STAGES) + 1024 + 256 + 1024 + 1024;
};

struct CmArgs {
  const float* lse2;   // [B, Hq, N]
  const float* vnorm;  // [B*N, Hkv] ||v|| per row and group (used when weight_vnorm)
  float* parts;        // [per][B][G][N]
  int B, N, Hq, Hkv, ld, n_kb, total, weight_vnorm;
  int causal;  // 0: bidirectional (every query block, no causal mask)
  const int* cu;  // packed sequences of different lengths: rows [cu[b], cu[b+1]); N = the longest
  const uint8_t* q_alive;  // masked mode: [B, N] flags, queries with 0 add nothing
  float scale_log2;
  int* status;
};

// 2^x with the MUFU approximation (flush-to-zero: soft-score terms below
// 2^-126 are negligible next to the column sums).
__device__ __forceinline__ float ex2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void cm_tile(int t, const CmArgs& a, int& b, int& g, int& hh, int& kb) {
  const int per = a.Hq / a.Hkv;
  const int inner = a.B * a.Hkv * per;
  kb = t / inner;  // large (early) key blocks first: they have the most query blocks
  int r = t % inner;
  hh = r % per;
  r /= per;
  g = r % a.Hkv;
  b = r / a.Hkv;
}

// Rows of sequence b: first packed row and length.
__device__ __forceinline__ void cm_seq(const CmArgs& a, int b, int& row0, int& n) {
  if (a.cu) {
    row0 = a.cu[b];
    n = a.cu[b + 1] - row0;
  } else {
    row0 = b * a.N;
    n = a.N;
  }
}

// Tile t holds keys of its sequence (a shorter sequence has fewer key blocks).
__device__ __forceinline__ bool cm_live(int t, const CmArgs& a) {
  int b, g, hh, kb, row0, n;
  cm_tile(t, a, b, g, hh, kb);
  cm_seq(a, b, row0, n);
  return kb * CM_BM < n;
}

// The next tile of this CTA at or after t that holds keys (a.total if none).
__device__ __forceinline__ int cm_next(int t, const CmArgs& a) {
  while (t < a.total && !cm_live(t, a)) t += gridDim.x;
  return t < a.total ? t : a.total;
}

template <int HD>
__global__ void __launch_bounds__(CM_THREADS, 2)
    colmass_tc_kernel(const __grid_constant__ CUtensorMap tm, const CmArgs a) {
  using C = CmCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = smem;                         // [2] K tiles
  uint8_t* sQ = smem + 2 * C::TILE_BYTES;      // [STAGES] Q tiles
  uint8_t* tail = smem + C::TILE_BYTES * (2 + CM_STAGES);
  uint64_t* full = reinterpret_cast<uint64_t*>(tail);  // [STAGES]
  uint64_t* empty = full + CM_STAGES;                  // [STAGES]
  uint64_t* kfull = empty + CM_STAGES;                 // [2] K tile loaded
  uint64_t* kempty = kfull + 2;                        // [2] K tile no longer read by MMAs
  uint64_t* acc_full = kempty + 2;                     // [2]
  uint64_t* acc_empty = acc_full + 2;                  // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* s_lse = reinterpret_cast<float*>(tail + 256);          // [2][128]
  float* s_half = reinterpret_cast<float*>(tail + 256 + 1024);  // [128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < CM_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kfull[i], 1);
      mbar_init(&kempty[i], 1);
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], CM_EPI_WARPS);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) prefetch_tmap(&tm);
  if (warp == 1) tmem_alloc(tmem_slot, 2 * CM_BN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0, tiles = 0, issued_last = 0;
      bool ok = true;
      for (int t = cm_next(blockIdx.x, a); t < a.total && ok; t = cm_next(t + gridDim.x, a), ++tiles) {
        int b, g, hh, kb, row0, n_b;
        cm_tile(t, a, b, g, hh, kb);
        cm_seq(a, b, row0, n_b);
        const int n_qb = (n_b + CM_BN - 1) / CM_BN;
        const int h = g * (a.Hq / a.Hkv) + hh;
        // K tile (two buffers): wait until the MMAs of two tiles ago are done with it
        const int kbuf = tiles & 1;
        if (!mbar_wait_ab(&kempty[kbuf], ((tiles >> 1) & 1) ^ 1, a.status, abort_flag)) break;
        mbar_arrive_expect_tx(&kfull[kbuf], C::TILE_BYTES);
        for (int c = 0; c < C::CHUNKS; ++c)
          tma_load_2d(sK + kbuf * C::TILE_BYTES + c * (C::TILE_BYTES / C::CHUNKS), &tm,
                      (a.Hq + g) * HD + c * 64, row0 + kb * CM_BM, &kfull[kbuf]);
        for (int qb = a.causal ? kb : 0; qb < n_qb; ++qb, ++it) {
          const int s = it % CM_STAGES;
          const uint32_t ph = (it / CM_STAGES) & 1;
          if (!mbar_wait_ab(&empty[s], ph ^ 1, a.status, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], C::TILE_BYTES);
          uint8_t* dst = sQ + s * C::TILE_BYTES;
          for (int c = 0; c < C::CHUNKS; ++c)
            tma_load_2d(dst + c * (C::TILE_BYTES / C::CHUNKS), &tm, h * HD + c * 64,
                        row0 + qb * CM_BN, &full[s]);
          issued_last = it + 1;
        }
      }
      if (!ok || *abort_flag) {
        for (uint32_t j = issued_last; j > 0 && j + CM_STAGES > issued_last; --j) {
          const uint32_t q = j - 1;
          mbar_wait(&full[q % CM_STAGES], (q / CM_STAGES) & 1, nullptr);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(CM_BM, CM_BN);
      uint32_t it = 0, tiles = 0;
      int i = 0;
      bool ok = true;
      for (int t = cm_next(blockIdx.x, a); t < a.total && ok; t = cm_next(t + gridDim.x, a), ++tiles) {
        int b, g, hh, kb, row0, n_b;
        cm_tile(t, a, b, g, hh, kb);
        cm_seq(a, b, row0, n_b);
        const int n_qb = (n_b + CM_BN - 1) / CM_BN;
        const int kbuf = tiles & 1;
        if (!mbar_wait_ab(&kfull[kbuf], (tiles >> 1) & 1, a.status, abort_flag)) break;
        tc_fence_after();
        const uint32_t k_base = smem_u32(sK + kbuf * C::TILE_BYTES);
        for (int qb = a.causal ? kb : 0; qb < n_qb; ++qb, ++it, ++i) {
          const int ab = i & 1;
          const uint32_t use = static_cast<uint32_t>(i >> 1);
          if (!mbar_wait_ab(&acc_empty[ab], (use & 1) ^ 1, a.status, abort_flag)) {
            ok = false;
            break;
          }
          const int s = it % CM_STAGES;
          const uint32_t ph = (it / CM_STAGES) & 1;
          if (!mbar_wait_ab(&full[s], ph, a.status, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t q_base = smem_u32(sQ + s * C::TILE_BYTES);
          const uint32_t d_tmem = tmem + static_cast<uint32_t>(ab * CM_BN);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t off = (kk / 4) * (C::TILE_BYTES / C::CHUNKS) + (kk % 4) * 32;
            tc_mma_bf16(d_tmem, sdesc_sw128(k_base + off), sdesc_sw128(q_base + off), idesc,
                        kk > 0 ? 1u : 0u);
          }
          tc_commit(&empty[s]);
          tc_commit(&acc_full[ab]);
        }
        tc_commit(&kempty[kbuf]);  // the K tile is free once these MMAs finish
      }
    }
    __syncwarp();
  } else {
    // Epilogue: 8 warps; quadrant = TMEM lanes, half = which 64 query columns.
    const int ew = warp - 2;
    const int quad = warp & 3, half = ew / 4;
    const int krow = quad * 32 + lane;  // key within the tile
    const int et = ew * 32 + lane;      // 0..255: loader of one normaliser
    // fetch the normalisers of step (t, qb) into s_lse[buf]
    auto fetch = [&](int t, int qb, int buf) {
      if (et < CM_BN) {
        int b, g, hh, kb, row0, n_b;
        cm_tile(t, a, b, g, hh, kb);
        cm_seq(a, b, row0, n_b);
        const int h = g * (a.Hq / a.Hkv) + hh;
        const int q = qb * CM_BN + et;
        float* dst = s_lse + buf * CM_BN + et;
        if (q < n_b && a.q_alive != nullptr && a.q_alive[static_cast<size_t>(b) * a.N + q] == 0) {
          *dst = INFINITY;  // exp2(s * c - inf) = 0: a hidden query contributes nothing
        } else if (q < n_b) {
          asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)),
                       "l"(a.lse2 + (static_cast<size_t>(b) * a.Hq + h) * a.N + q)
                       : "memory");
        } else {
          *dst = 0.f;
        }
      }
      cp_async_commit();
    };
    int i = 0;
    bool ok = true;
    const int t_first = cm_next(blockIdx.x, a);
    if (t_first < a.total) {
      int b, g, hh, kb;
      cm_tile(t_first, a, b, g, hh, kb);
      fetch(t_first, a.causal ? kb : 0, 0);
    }
    for (int t = t_first; t < a.total; t = cm_next(t + gridDim.x, a)) {
      int b, g, hh, kb, row0, n_b;
      cm_tile(t, a, b, g, hh, kb);
      cm_seq(a, b, row0, n_b);
      const int n_qb = (n_b + CM_BN - 1) / CM_BN;
      const int key = kb * CM_BM + krow;
      float acc = 0.f;
      for (int qb = a.causal ? kb : 0; qb < n_qb; ++qb, ++i) {
        const int ab = i & 1;
        const uint32_t use = static_cast<uint32_t>(i >> 1);
        cp_async_wait<0>();
        // this step's normalisers are in s_lse[ab]; every warp is done with step i-1
        asm volatile("bar.sync 1, %0;" ::"n"(CM_EPI_WARPS * 32) : "memory");
        if (qb + 1 < n_qb) {
          fetch(t, qb + 1, ab ^ 1);
        } else {
          const int tn = cm_next(t + gridDim.x, a);
          if (tn < a.total) {
            int b2, g2, hh2, kb2;
            cm_tile(tn, a, b2, g2, hh2, kb2);
            fetch(tn, a.causal ? kb2 : 0, ab ^ 1);
          }
        }
        const float* L = s_lse + ab * CM_BN;
        ok = ok && __all_sync(0xffffffffu, mbar_wait_ab(&acc_full[ab], use & 1, a.status, abort_flag));
        tc_fence_after();
        if (ok) {
          const uint32_t tbase = tmem + static_cast<uint32_t>(ab * CM_BN + half * 64) +
                                 (static_cast<uint32_t>(quad * 32) << 16);
#pragma unroll 1
          for (int c = 0; c < 64; c += 32) {
            uint32_t r[32];
            __syncwarp();
            tmem_ld16(tbase + c, *reinterpret_cast<uint32_t(*)[16]>(r));
            tmem_ld16(tbase + c + 16, *reinterpret_cast<uint32_t(*)[16]>(r + 16));
            tmem_ld_wait();
            const int qc0 = half * 64 + c;
            const int q0 = qb * CM_BN + qc0;
            if ((!a.causal || q0 > key) && q0 + 32 <= n_b) {  // whole chunk inside the mask
              // lse - s c for two columns in one packed FMA, then exp2 of its
              // negation (the same rounding as s c - lse), summed in pairs:
              // half the FMA-pipe instructions, which the MMA thread on the
              // same SMSP competes with for issue slots
              const uint64_t nc2 = f2pack(-a.scale_log2, -a.scale_log2);
              uint64_t acc2 = f2pack(0.f, 0.f);
#pragma unroll
              for (int e = 0; e < 32; e += 2) {
                const uint64_t u = ffma2(f2pack(__uint_as_float(r[e]), __uint_as_float(r[e + 1])), nc2,
                                         *reinterpret_cast<const uint64_t*>(L + qc0 + e));
                float u0, u1;
                f2unpack(u, u0, u1);
                acc2 = fadd2(acc2, f2pack(ex2_ftz(-u0), ex2_ftz(-u1)));
              }
              float a0, a1;
              f2unpack(acc2, a0, a1);
              acc += a0 + a1;
            } else {
#pragma unroll
              for (int e = 0; e < 32; ++e) {
                const int q = q0 + e;
                if ((!a.causal || q >= key) && q < n_b)
                  acc += ex2_ftz(__uint_as_float(r[e]) * a.scale_log2 - L[qc0 + e]);
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acc_empty[ab])) : "memory");
      }
      // add the two column halves (fixed order: half 0 + half 1)
      if (half == 1) s_half[krow] = acc;
      asm volatile("bar.sync 1, %0;" ::"n"(CM_EPI_WARPS * 32) : "memory");
      if (half == 0 && key < n_b) {
        float v = acc + s_half[krow];
        if (a.weight_vnorm) v *= a.vnorm[(static_cast<size_t>(row0) + key) * a.Hkv + g];
        a.parts[((static_cast<size_t>(hh) * a.B + b) * a.Hkv + g) * a.N + key] = v;
      }
      // s_half is rewritten only after the next tile's first barrier
    }
    cp_async_wait<0>();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * CM_BN);
  }
}

int cm_num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}

template <int HD>
cudaError_t run_cm(const CUtensorMap& tm, const CmArgs& a, int sms, cudaStream_t s) {
  using C = CmCfg<HD>;
  static OncePerDevice once;
  const cudaError_t attr_err = set_smem_limit_once(once, colmass_tc_kernel<HD>, static_cast<int>(C::SMEM));
  // Two CTAs per SM when their shared memory fits (hd 64): they hide each
  // other's epilogue latency (TMEM: 2 x 256 columns; registers: 2 x 320 x 96).
  constexpr int per_sm = 2 * (C::SMEM + 1024) <= 227 * 1024 ? 2 : 1;
  if (attr_err != cudaSuccess) return attr_err;
  const int cap = sms * per_sm;
  const int grid = a.total < cap ? a.total : cap;
  ZSAA_LAUNCH(colmass_tc_kernel<HD>, dim3(grid), dim3(CM_THREADS), C::SMEM, s, tm, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_colmass_tc(const void* qkv, const float* lse, const float* vnorm, int B, int N,
                              int Hq, int Hkv, int hd, float* parts, int* status, int* n_chunks,
                              int causal, cudaStream_t s, const int* cu, int rows,
                              const uint8_t* q_alive) {
  if (hd != 64 && hd != 128) return cudaErrorInvalidValue;
  const int ld = (Hq + 2 * Hkv) * hd;
  EncodeTiledFn enc = get_encode_tiled();
  if (enc == nullptr) return cudaErrorInvalidValue;
  CUtensorMap tm;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(ld),
                        cu ? static_cast<cuuint64_t>(rows) : static_cast<cuuint64_t>(B) * N};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(CM_BM)};
  cuuint32_t es[2] = {1, 1};
  if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(qkv), dims, strides, box, es,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  CmArgs a;
  a.lse2 = lse;
  a.vnorm = vnorm;
  a.parts = parts;
  a.B = B;
  a.N = N;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.ld = ld;
  a.n_kb = (N + CM_BM - 1) / CM_BM;
  a.total = a.n_kb * B * Hq;
  a.weight_vnorm = vnorm != nullptr;
  a.causal = causal;
  a.cu = cu;
  a.q_alive = q_alive;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  a.status = status;
  *n_chunks = Hq / Hkv;
  const int sms = cm_num_sms();
  return hd == 64 ? run_cm<64>(tm, a, sms, s) : run_cm<128>(tm, a, sms, s);
}

}  // namespace zsaa
