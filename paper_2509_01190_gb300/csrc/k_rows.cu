// Row-wise kernels of the pruned prefill: embedding gather, RMSNorm, row-norm
// scores of the isolated path (Sec. 3.3 with unit column mass), per-sequence
// top-k selection, row compaction, fp32 RoPE and the classifier head.  All are HBM-bound: one warp per row, 16-byte
// vector accesses, fp32 arithmetic.
#include "common.cuh"
#include "kernels.h"

namespace zsaa {

namespace {

constexpr int kWarpsPerBlock = 8;
// Rows of up to 32 * kMaxVecPerLane 16-byte vectors (d <= 4096 in bf16) are
// held in registers, a lane's vectors all in flight at once.
constexpr int kMaxVecPerLane = 16;

inline int row_blocks(int rows) { return (rows + kWarpsPerBlock - 1) / kWarpsPerBlock; }

// ---------------------------------------------------------------- embedding

// h[r, :] = E[tok[r], :], pos[r] = r mod L  (a row is d * elem bytes, copied as uint4)
// A token id outside [0, vocab) sets kStatusBadIndex and embeds row 0.
__global__ void embed_kernel(const uint4* __restrict__ E, const int32_t* __restrict__ tok, int rows,
                             int L, int vocab, int vec_per_row, uint4* __restrict__ h,
                             int32_t* __restrict__ pos, int* status) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  int t = tok[r];
  if (t < 0 || t >= vocab) {
    if (lane == 0 && status != nullptr) atomicOr(status, kStatusBadIndex);
    t = 0;
  }
  const uint4* src = E + static_cast<size_t>(t) * vec_per_row;
  uint4* dst = h + static_cast<size_t>(r) * vec_per_row;
  for (int v = lane; v < vec_per_row; v += 32) dst[v] = __ldg(src + v);
  if (lane == 0) pos[r] = r % L;
}

// ---------------------------------------------------------------- RMSNorm

// The norm weights of a row (n16 16-byte vectors) are never written by a
// kernel: a warp asks L2 for them, one 128-byte line per lane, before it waits
// for the previous kernel, so they are not a round trip on the row's chain of
// dependent loads.
__device__ __forceinline__ void prefetch_norm_weights(const uint4* w, int n16, int lane) {
  for (int line = lane; line * 8 < n16; line += 32)
    asm volatile("prefetch.global.L2 [%0];" ::"l"(w + line * 8));
}

template <typename T>
__global__ void rmsnorm_kernel(const T* __restrict__ h, const T* __restrict__ w, int rows, int d,
                               float eps, T* __restrict__ x) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const T* hr = h + static_cast<size_t>(r) * d;
  T* xr = x + static_cast<size_t>(r) * d;
  float ss = 0.f;
  for (int i = lane; i < d; i += 32) {
    float v = to_f(hr[i]);
    ss += v * v;
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(d) + eps);
  for (int i = lane; i < d; i += 32) xr[i] = from_f<T>(to_f(hr[i]) * inv * to_f(w[i]));
}

// The norm weights (vec 16-byte vectors, never written by a kernel) staged in
// the block's shared memory before the wait for the previous kernel: every
// warp of the block reads them there instead of from L2.
__device__ __forceinline__ void stage_norm_weights(const uint4* __restrict__ w, int vec, uint4* sw) {
  for (int v = threadIdx.x; v < vec; v += blockDim.x) sw[v] = __ldg(w + v);
  __syncthreads();
}

// bf16 rows of at most 32 * kMaxVecPerLane vectors: one warp per row, the row
// loaded into registers once (every load of a lane in flight together), its
// sum of squares, then x = h / rms * w with the weights from shared memory.
__global__ void rmsnorm_bf16_reg_kernel(const uint4* __restrict__ h, const uint4* __restrict__ w,
                                        int rows, int vec, float eps, uint4* __restrict__ x) {
  extern __shared__ uint4 sw[];
  pdl_trigger();
  stage_norm_weights(w, vec, sw);
  pdl_wait();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const uint4* hr = h + static_cast<size_t>(r) * vec;
  uint4* xr = x + static_cast<size_t>(r) * vec;
  uint4 u[kMaxVecPerLane];
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < kMaxVecPerLane; ++q) {
    const int v = lane + 32 * q;
    if (v < vec) u[q] = hr[v];
  }
#pragma unroll
  for (int q = 0; q < kMaxVecPerLane; ++q) {
    const int v = lane + 32 * q;
    if (v < vec) {
      const uint32_t e4[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = bf16lo(e4[e]), c = bf16hi(e4[e]);
        ss += a * a + c * c;
      }
    }
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(vec * 8) + eps);
#pragma unroll
  for (int q = 0; q < kMaxVecPerLane; ++q) {
    const int v = lane + 32 * q;
    if (v < vec) {
      const uint4 wv = sw[v];
      const uint32_t e4[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
      const uint32_t w4[4] = {wv.x, wv.y, wv.z, wv.w};
      uint32_t o[4];
#pragma unroll
      for (int e = 0; e < 4; ++e)
        o[e] = pack_bf16x2(bf16lo(e4[e]) * inv * bf16lo(w4[e]), bf16hi(e4[e]) * inv * bf16hi(w4[e]));
      xr[v] = make_uint4(o[0], o[1], o[2], o[3]);
    }
  }
}

// bf16 rows, 8 elements per 16-byte vector (any length).
__global__ void rmsnorm_bf16_vec_kernel(const uint4* __restrict__ h, const uint4* __restrict__ w,
                                        int rows, int vec_per_row, float eps,
                                        uint4* __restrict__ x) {
  pdl_trigger();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < 32) prefetch_norm_weights(w, vec_per_row, lane);
  pdl_wait();
  if (r >= rows) return;
  const uint4* hr = h + static_cast<size_t>(r) * vec_per_row;
  uint4* xr = x + static_cast<size_t>(r) * vec_per_row;
  float ss = 0.f;
  for (int v = lane; v < vec_per_row; v += 32) {
    uint4 u = hr[v];
    const uint32_t p[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float a = bf16lo(p[q]), b = bf16hi(p[q]);
      ss += a * a + b * b;
    }
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(vec_per_row * 8) + eps);
  for (int v = lane; v < vec_per_row; v += 32) {
    uint4 u = hr[v], wv = __ldg(w + v);
    const uint32_t p[4] = {u.x, u.y, u.z, u.w};
    const uint32_t q4[4] = {wv.x, wv.y, wv.z, wv.w};
    uint32_t o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q)
      o[q] = pack_bf16x2(bf16lo(p[q]) * inv * bf16lo(q4[q]), bf16hi(p[q]) * inv * bf16hi(q4[q]));
    xr[v] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// ---------------------------------------------------------------- scores

// s[r] = ||h[r, :]||_2 for bf16 rows (the score with unit column mass, one group).
template <int UNROLL>
__global__ void row_norm_bf16_kernel(const uint4* __restrict__ h, int rows, int vec_per_row,
                                     float* __restrict__ s) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const uint4* hr = h + static_cast<size_t>(r) * vec_per_row;
  float ss = 0.f;
  int v = lane;
  for (; v + 32 * (UNROLL - 1) < vec_per_row; v += 32 * UNROLL) {
    uint4 u[UNROLL];
#pragma unroll
    for (int q = 0; q < UNROLL; ++q) u[q] = __ldcs(hr + v + 32 * q);
#pragma unroll
    for (int q = 0; q < UNROLL; ++q) {
      const uint32_t p[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float a = bf16lo(p[e]), b = bf16hi(p[e]);
        ss = fmaf(a, a, ss);
        ss = fmaf(b, b, ss);
      }
    }
  }
  for (; v < vec_per_row; v += 32) {
    uint4 u = __ldcs(hr + v);
    const uint32_t p[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float a = bf16lo(p[e]), b = bf16hi(p[e]);
      ss = fmaf(a, a, ss);
      ss = fmaf(b, b, ss);
    }
  }
  ss = warp_sum(ss);
  if (lane == 0) s[r] = sqrtf(ss);
}

__global__ void row_norm_f32_kernel(const float* __restrict__ h, int rows, int d,
                                    float* __restrict__ s) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const float* hr = h + static_cast<size_t>(r) * d;
  float ss = 0.f;
  for (int i = lane; i < d; i += 32) ss = fmaf(hr[i], hr[i], ss);
  ss = warp_sum(ss);
  if (lane == 0) s[r] = sqrtf(ss);
}

// ---------------------------------------------------------------- top-k select

// Order-preserving map float -> uint32 (larger float -> larger key).  NaN maps
// to 0, below every number; -0 is folded onto +0.
__device__ __forceinline__ uint32_t order_key(float f) {
  uint32_t u = __float_as_uint(f);
  if (f != f) return 0u;
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// One block per sequence, of THREADS threads (256 to 1024, by the sequence
// length: the selection is a chain of block-wide barriers, which cost less in
// a smaller block, and a 1024-thread block left most of its threads idle on
// the few hundred kept rows of the deep pruned layers).  Radix select (4 passes of 8 bits) finds the key T of
// the need-th best candidate and how many candidates equal to T are taken;
// then an index-ordered ballot/prefix scan writes the kept indices ascending.
// Up to 256 candidates without marks take a shorter route to the same set:
// each thread counts its candidate's rank against all others.
// Ties (equal keys) keep lower indices first.  With force_last the last index
// is kept and the other k-1 come from indices [0, N-1).
// FROM_PARTS: the scores are first summed from column-mass partials
// parts[qc][b][g][j] (n_qc chunks, G groups) into shared memory (and copied to
// scores_out when it is not null); otherwise they are read from `scores`.
template <bool FROM_PARTS, int THREADS>
__global__ void __launch_bounds__(THREADS)
    select_topk_kernel(const float* __restrict__ scores, int Ns, int ks, int force_last,
                       int32_t* __restrict__ idx_out, const float* __restrict__ parts, int n_qc,
                       int B, int G, float* __restrict__ scores_out, const int* __restrict__ cu_in,
                       const int* __restrict__ cu_out, uint8_t* __restrict__ alive) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  // fixed length: N = Ns rows in, k = ks kept per sequence; variable length
  // (FROM_PARTS only): this sequence's counts from the packed row offsets,
  // partials still at stride Ns (the longest sequence)
  const int N = cu_in ? cu_in[b + 1] - cu_in[b] : Ns;
  const int k = cu_out ? cu_out[b + 1] - cu_out[b] : ks;
  const size_t sc_row0 = cu_in ? static_cast<size_t>(cu_in[b]) : static_cast<size_t>(b) * Ns;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int nwarps = THREADS / 32;
  extern __shared__ float sscore[];
  const float* s = scores + static_cast<size_t>(b) * N;
  if (FROM_PARTS) {
    // Partial t = qc * G + g lives at parts + qc * plane + (b * G + g) * Ns;
    // the sum runs over t in increasing order.  The loads are issued kSumBatch
    // at a time, ahead of their adds, so the chain waits for L2 once per
    // batch instead of once per partial (the adds keep their order).
    constexpr int kSumBatch = 16;
    const size_t plane = static_cast<size_t>(B) * G * Ns;
    const int np = n_qc * G;
    const float* pb = parts + static_cast<size_t>(b) * G * Ns;
    for (int j = tid; j < N; j += THREADS) {
      float acc = 0.f;
      const float* pj = pb + j;
      int t = 0, g = 0;
      size_t qoff = 0;  // qc * plane of partial t = qc * G + g
      for (; t + kSumBatch <= np; t += kSumBatch) {
        float v[kSumBatch];
#pragma unroll
        for (int u = 0; u < kSumBatch; ++u) {
          v[u] = pj[qoff + static_cast<size_t>(g) * Ns];
          if (++g == G) {
            g = 0;
            qoff += plane;
          }
        }
#pragma unroll
        for (int u = 0; u < kSumBatch; ++u) acc += v[u];
      }
      for (; t < np; ++t) {
        acc += pj[qoff + static_cast<size_t>(g) * Ns];
        if (++g == G) {
          g = 0;
          qoff += plane;
        }
      }
      sscore[j] = acc;
      if (scores_out != nullptr) scores_out[sc_row0 + j] = acc;
    }
    __syncthreads();
    s = sscore;
  }
  int32_t* out = idx_out + (cu_out ? static_cast<size_t>(cu_out[b]) : static_cast<size_t>(b) * k);
  // masked mode (Appendix B, fixed length): rows are never removed; the
  // candidates are the rows still unmarked, and the flags are updated here
  uint8_t* al = alive ? alive + static_cast<size_t>(b) * Ns : nullptr;
  const int n_cand = force_last ? N - 1 : N;
  const int need = force_last ? k - 1 : k;

  __shared__ __align__(16) uint32_t hist[256];
  __shared__ uint32_t sh_digit, sh_remaining;
  __shared__ int wgt[nwarps], weq[nwarps];
  __shared__ int tile_gt, tile_eq;
  const uint32_t lt_mask = (1u << lane) - 1u;

  if (THREADS == 256 && al == nullptr && n_cand <= THREADS) {
    // Short sequence, one candidate per thread: count the candidates ahead of
    // candidate j in (key descending, index ascending) order directly.  Rank <
    // need is the radix path's kept set (every key above the threshold, then
    // equal keys lowest index first), without its four barrier-bound passes.
    uint32_t* skey = hist;  // THREADS keys; the padding (key 0) never counts
    const int j = tid;
    const uint32_t kj = j < n_cand ? order_key(s[j]) : 0u;
    skey[j] = kj;
    __syncthreads();
    int rank = 0;
    const int n4 = (n_cand + 3) & ~3;
    for (int i0 = 0; i0 < n4; i0 += 4) {
      const uint4 k4 = *reinterpret_cast<const uint4*>(skey + i0);
      rank += (k4.x > kj) + (k4.x == kj && i0 < j);
      rank += (k4.y > kj) + (k4.y == kj && i0 + 1 < j);
      rank += (k4.z > kj) + (k4.z == kj && i0 + 2 < j);
      rank += (k4.w > kj) + (k4.w == kj && i0 + 3 < j);
    }
    const bool keep = j < n_cand && rank < need;
    const uint32_t bk = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) wgt[warp] = __popc(bk);
    __syncthreads();
    int before = __popc(bk & lt_mask);
    for (int w = 0; w < warp; ++w) before += wgt[w];
    if (keep) out[before] = j;
    if (force_last && tid == 0) out[k - 1] = N - 1;
    return;
  }

  uint32_t prefix = 0, mask = 0, remaining = static_cast<uint32_t>(need);
  if (need > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 256; i += THREADS) hist[i] = 0;
      __syncthreads();
      for (int j = tid; j < n_cand; j += THREADS) {
        if (al != nullptr && al[j] == 0) continue;  // masked mode: only unmarked rows compete
        const uint32_t key = order_key(s[j]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        uint32_t c[8], local = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          c[q] = hist[lane * 8 + q];
          local += c[q];
        }
        uint32_t suf = local;  // inclusive suffix sum over lanes
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          uint32_t v = __shfl_down_sync(0xffffffffu, suf, o);
          if (lane + o < 32) suf += v;
        }
        uint32_t acc = suf - local;  // candidates in bins of higher lanes
#pragma unroll
        for (int q = 7; q >= 0; --q) {
          if (acc < remaining && acc + c[q] >= remaining) {
            sh_digit = static_cast<uint32_t>(lane * 8 + q);
            sh_remaining = remaining - acc;
          }
          acc += c[q];
        }
      }
      __syncthreads();
      prefix |= sh_digit << shift;
      mask |= 255u << shift;
      remaining = sh_remaining;
      __syncthreads();
    }
  }
  const uint32_t T = prefix;
  int base_gt = 0, base_eq = 0;
  for (int j0 = 0; j0 < n_cand && need > 0; j0 += THREADS) {
    const int j = j0 + tid;
    const bool in = j < n_cand && (al == nullptr || al[j] != 0);
    const uint32_t key = in ? order_key(s[j]) : 0u;
    const bool gt = in && key > T;
    const bool eq = in && key == T;
    const uint32_t bgt = __ballot_sync(0xffffffffu, gt), beq = __ballot_sync(0xffffffffu, eq);
    if (lane == 0) {
      wgt[warp] = __popc(bgt);
      weq[warp] = __popc(beq);
    }
    __syncthreads();
    if (warp == 0) {  // exclusive scan of the per-warp counts
      int a = lane < nwarps ? wgt[lane] : 0, e = lane < nwarps ? weq[lane] : 0;
      int ia = a, ie = e;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int va = __shfl_up_sync(0xffffffffu, ia, o), ve = __shfl_up_sync(0xffffffffu, ie, o);
        if (lane >= o) {
          ia += va;
          ie += ve;
        }
      }
      if (lane < nwarps) {
        wgt[lane] = ia - a;
        weq[lane] = ie - e;
      }
      if (lane == 31) {
        tile_gt = ia;
        tile_eq = ie;
      }
    }
    __syncthreads();
    const int gt_before = base_gt + wgt[warp] + __popc(bgt & lt_mask);
    const int eq_before = base_eq + weq[warp] + __popc(beq & lt_mask);
    const int rem = static_cast<int>(remaining);
    if (gt || (eq && eq_before < rem)) out[gt_before + min(eq_before, rem)] = j;
    base_gt += tile_gt;
    base_eq += tile_eq;
    __syncthreads();
  }
  if (force_last && tid == 0) out[k - 1] = N - 1;
  if (al != nullptr) {  // the kept rows stay unmarked, every other row is marked
    __syncthreads();
    for (int j = tid; j < N; j += THREADS) al[j] = 0;
    __syncthreads();
    for (int r = tid; r < k; r += THREADS) al[out[r]] = 1;
  }
}

// Masked mode with given kept positions: flags[b, :] = 0, then 1 at idx[b, :k].
__global__ void flags_from_idx_kernel(const int32_t* __restrict__ idx, int N, int k,
                                      uint8_t* __restrict__ flags, int* status) {
  pdl_trigger();
  pdl_wait();
  uint8_t* f = flags + static_cast<size_t>(blockIdx.x) * N;
  for (int j = threadIdx.x; j < N; j += blockDim.x) f[j] = 0;
  __syncthreads();
  for (int r = threadIdx.x; r < k; r += blockDim.x) {
    const int j = idx[static_cast<size_t>(blockIdx.x) * k + r];
    if (j >= 0 && j < N)
      f[j] = 1;
    else if (status != nullptr)
      atomicOr(status, kStatusBadIndex);
  }
}

// ---------------------------------------------------------------- gather

// dst[b*k + r, :] = src[b*N + idx[b*k + r], :]; pos_out likewise.  One warp per row.
// An index outside [0, N) sets kStatusBadIndex and copies row 0 instead.
template <int UNROLL>
__global__ void gather_rows_kernel(const uint4* __restrict__ src, int N, int k, int vec_per_row,
                                   const int32_t* __restrict__ idx, uint4* __restrict__ dst,
                                   const int32_t* __restrict__ pos_in, int32_t* __restrict__ pos_out,
                                   int total, int* status) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= total) return;
  const int b = r / k;
  int j = idx[r];
  if (j < 0 || j >= N) {
    if (lane == 0 && status != nullptr) atomicOr(status, kStatusBadIndex);
    j = 0;
  }
  const size_t srow = static_cast<size_t>(b) * N + j;
  const uint4* s = src + srow * vec_per_row;
  uint4* d = dst + static_cast<size_t>(r) * vec_per_row;
  int v = lane;
  for (; v + 32 * (UNROLL - 1) < vec_per_row; v += 32 * UNROLL) {
    uint4 u[UNROLL];
#pragma unroll
    for (int q = 0; q < UNROLL; ++q) u[q] = s[v + 32 * q];
#pragma unroll
    for (int q = 0; q < UNROLL; ++q) __stcs(d + v + 32 * q, u[q]);
  }
  for (; v < vec_per_row; v += 32) __stcs(d + v, s[v]);
  if (pos_out != nullptr && lane == 0) pos_out[r] = pos_in[srow];
}

// ---------------------------------------------------------------- row copy + RMSNorm

// Copies source rows into the residual buffer and writes their RMSNorm, for
// bf16 rows of d = 8 * vec elements (vec <= 32 * kMaxVecPerLane):
//   embedding (idx == nullptr): source row tok[r] of E, pos_out[r] = r mod L;
//   compaction: source row b*N + idx[r] of h (b = r / k), pos_out[r] =
//     pos_in[that row] -- the kept rows of the previous layer, already normed
//     for the next layer's attention.
// An index outside its range sets kStatusBadIndex and copies row 0.
__global__ void rows_norm_bf16_kernel(const uint4* __restrict__ src, const int32_t* __restrict__ tok,
                                      int vocab, int L, const int32_t* __restrict__ idx, int N,
                                      int k, const int32_t* __restrict__ pos_in, int rows, int vec,
                                      const uint4* __restrict__ w, float eps,
                                      uint4* __restrict__ h_out, uint4* __restrict__ x_out,
                                      int32_t* __restrict__ pos_out, int* status,
                                      const int* __restrict__ cu_src, const int* __restrict__ cu_dst,
                                      int nseq) {
  extern __shared__ uint4 sw[];
  pdl_trigger();
  const int r = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  stage_norm_weights(w, vec, sw);
  pdl_wait();
  if (r >= rows) return;
  size_t srow;
  int p;
  if (idx == nullptr) {
    int t = tok[r];
    if (t < 0 || t >= vocab) {
      if (lane == 0 && status != nullptr) atomicOr(status, kStatusBadIndex);
      t = 0;
    }
    srow = static_cast<size_t>(t);
    p = cu_dst ? r - __ldg(cu_dst + seq_of_row(cu_dst, nseq, r)) : r % L;
  } else {
    int b, n_b;
    size_t row0;
    if (cu_dst) {  // packed sequences of different lengths
      b = seq_of_row(cu_dst, nseq, r);
      row0 = static_cast<size_t>(__ldg(cu_src + b));
      n_b = __ldg(cu_src + b + 1) - __ldg(cu_src + b);
    } else {
      b = r / k;
      row0 = static_cast<size_t>(b) * N;
      n_b = N;
    }
    int j = idx[r];
    if (j < 0 || j >= n_b) {
      if (lane == 0 && status != nullptr) atomicOr(status, kStatusBadIndex);
      j = 0;
    }
    srow = row0 + j;
    p = pos_in[srow];
  }
  const uint4* sr = src + srow * vec;
  uint4* hr = h_out + static_cast<size_t>(r) * vec;
  uint4* xr = x_out + static_cast<size_t>(r) * vec;
  uint4 u[kMaxVecPerLane];
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < kMaxVecPerLane; ++q) {
    const int v = lane + 32 * q;
    if (v < vec) {
      u[q] = sr[v];
      hr[v] = u[q];
      const uint32_t e4[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = bf16lo(e4[e]), c = bf16hi(e4[e]);
        ss += a * a + c * c;
      }
    }
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(vec * 8) + eps);
#pragma unroll
  for (int q = 0; q < kMaxVecPerLane; ++q) {
    const int v = lane + 32 * q;
    if (v < vec) {
      const uint4 wv = sw[v];
      const uint32_t e4[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
      const uint32_t w4[4] = {wv.x, wv.y, wv.z, wv.w};
      uint32_t o[4];
#pragma unroll
      for (int e = 0; e < 4; ++e)
        o[e] = pack_bf16x2(bf16lo(e4[e]) * inv * bf16lo(w4[e]), bf16hi(e4[e]) * inv * bf16hi(w4[e]));
      xr[v] = make_uint4(o[0], o[1], o[2], o[3]);
    }
  }
  if (lane == 0) pos_out[r] = p;
}

// ---------------------------------------------------------------- RoPE (fp32 path)

// Rotate pairs (c, c + hd/2) of every head in columns [0, rope_cols) of each row.
__global__ void rope_f32_kernel(float* __restrict__ qkv, int rows, int ld, int rope_cols, int hd,
                                const int32_t* __restrict__ pos, const float* __restrict__ cos_t,
                                const float* __restrict__ sin_t) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.y;
  const int half = hd / 2;
  const int pairs = rope_cols / 2;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= rows || t >= pairs) return;
  const int head = t / half, c = t % half;
  const int p = pos[r];
  float* x = qkv + static_cast<size_t>(r) * ld + head * hd;
  const float cs = cos_t[static_cast<size_t>(p) * half + c];
  const float sn = sin_t[static_cast<size_t>(p) * half + c];
  const float x1 = x[c], x2 = x[c + half];
  x[c] = x1 * cs - x2 * sn;
  x[c + half] = x2 * cs + x1 * sn;
}

// ---------------------------------------------------------------- classifier head

// out[b, c] = sum_i xn[i] * W[c, i], xn = storage(rmsnorm(h[b, N-1]) * w)
template <typename T>
__global__ void cls_head_kernel(const T* __restrict__ h, int N, int d,
                                const T* __restrict__ norm_w, float eps, const T* __restrict__ W,
                                int n_classes, float* __restrict__ out, const int* __restrict__ cu) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float xs[];  // d floats
  __shared__ float red[32];
  const int b = blockIdx.x;
  const size_t last = cu ? static_cast<size_t>(cu[b + 1] - 1) : static_cast<size_t>(b) * N + (N - 1);
  const T* row = h + last * d;
  float ss = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    float v = to_f(row[i]);
    ss += v * v;
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < blockDim.x / 32 ? red[threadIdx.x] : 0.f;
    v = warp_sum(v);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = rsqrtf(red[0] / static_cast<float>(d) + eps);
  for (int i = threadIdx.x; i < d; i += blockDim.x)
    xs[i] = to_f(from_f<T>(to_f(row[i]) * inv * to_f(norm_w[i])));
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int c = warp; c < n_classes; c += blockDim.x / 32) {
    const T* wr = W + static_cast<size_t>(c) * d;
    float acc = 0.f;
    for (int i = lane; i < d; i += 32) acc = fmaf(xs[i], to_f(wr[i]), acc);
    acc = warp_sum(acc);
    if (lane == 0) out[static_cast<size_t>(b) * n_classes + c] = acc;
  }
}

}  // namespace

cudaError_t launch_embed(int dtype, const void* E, const int32_t* tok, int rows, int L, int vocab,
                         int d, void* h, int32_t* pos, int* status, cudaStream_t s) {
  const int esz = dtype == ZSAA_BF16 ? 2 : 4;
  const int vec = d * esz / 16;
  ZSAA_LAUNCH(embed_kernel, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock), 0, s, 
      static_cast<const uint4*>(E), tok, rows, L, vocab, vec, static_cast<uint4*>(h), pos, status);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(int dtype, const void* h, const void* w, int rows, int d, float eps,
                           void* x, cudaStream_t s) {
  if (dtype == ZSAA_BF16 && d % 8 == 0 && d / 8 <= 32 * kMaxVecPerLane) {
    ZSAA_LAUNCH(rmsnorm_bf16_reg_kernel, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock),
                static_cast<size_t>(d / 8) * 16, s, static_cast<const uint4*>(h), static_cast<const uint4*>(w),
                rows, d / 8, eps, static_cast<uint4*>(x));
  } else if (dtype == ZSAA_BF16 && d % 8 == 0) {
    ZSAA_LAUNCH(rmsnorm_bf16_vec_kernel, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock), 0, s, 
        static_cast<const uint4*>(h), static_cast<const uint4*>(w), rows, d / 8, eps,
        static_cast<uint4*>(x));
  } else if (dtype == ZSAA_BF16) {
    ZSAA_LAUNCH(rmsnorm_kernel<bf16>, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock), 0, s, 
        static_cast<const bf16*>(h), static_cast<const bf16*>(w), rows, d, eps,
        static_cast<bf16*>(x));
  } else {
    ZSAA_LAUNCH(rmsnorm_kernel<float>, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock), 0, s, 
        static_cast<const float*>(h), static_cast<const float*>(w), rows, d, eps,
        static_cast<float*>(x));
  }
  return cudaGetLastError();
}

cudaError_t launch_row_norm(int dtype, const void* h, int rows, int d, float* scores,
                            cudaStream_t s) {
  if (dtype == ZSAA_BF16) {
    ZSAA_LAUNCH(row_norm_bf16_kernel<8>, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock), 0, s, 
        static_cast<const uint4*>(h), rows, d / 8, scores);
  } else {
    ZSAA_LAUNCH(row_norm_f32_kernel, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock), 0, s, 
        static_cast<const float*>(h), rows, d, scores);
  }
  return cudaGetLastError();
}

// Threads of a selection block for sequences of up to N rows.
inline int sel_threads(int N) { return N <= 512 ? 256 : (N <= 2048 ? 512 : 1024); }

template <bool FROM_PARTS, int T>
cudaError_t launch_select_t(const float* scores, const float* parts, int n_qc, int B, int G, int N, int k,
                            int force_last, int32_t* idx, float* scores_out, size_t smem, cudaStream_t s,
                            const int* cu_in, const int* cu_out, uint8_t* alive) {
  if (FROM_PARTS) {
    static OncePerDevice once;
    const cudaError_t attr = set_smem_limit_once(once, select_topk_kernel<true, T>,
                                                 static_cast<int>(kSelectPartsMaxN * sizeof(float)));
    if (attr != cudaSuccess) return attr;
  }
  ZSAA_LAUNCH(select_topk_kernel<FROM_PARTS, T>, dim3(B), dim3(T), smem, s, scores, N, k, force_last, idx, parts,
              n_qc, B, G, scores_out, cu_in, cu_out, alive);
  return cudaGetLastError();
}

template <bool FROM_PARTS>
cudaError_t launch_select_any(const float* scores, const float* parts, int n_qc, int B, int G, int N, int k,
                              int force_last, int32_t* idx, float* scores_out, size_t smem, cudaStream_t s,
                              const int* cu_in, const int* cu_out, uint8_t* alive) {
  switch (sel_threads(N)) {
    case 256:
      return launch_select_t<FROM_PARTS, 256>(scores, parts, n_qc, B, G, N, k, force_last, idx, scores_out, smem,
                                              s, cu_in, cu_out, alive);
    case 512:
      return launch_select_t<FROM_PARTS, 512>(scores, parts, n_qc, B, G, N, k, force_last, idx, scores_out, smem,
                                              s, cu_in, cu_out, alive);
    default:
      return launch_select_t<FROM_PARTS, 1024>(scores, parts, n_qc, B, G, N, k, force_last, idx, scores_out,
                                               smem, s, cu_in, cu_out, alive);
  }
}

cudaError_t launch_select(const float* scores, int B, int N, int k, int force_last, int32_t* idx,
                          cudaStream_t s) {
  return launch_select_any<false>(scores, nullptr, 0, B, 0, N, k, force_last, idx, nullptr, 0, s, nullptr, nullptr,
                                  nullptr);
}

cudaError_t launch_select_parts(const float* parts, int n_qc, int B, int G, int N, int k,
                                int force_last, int32_t* idx, float* scores_out, cudaStream_t s,
                                const int* cu_in, const int* cu_out, uint8_t* alive) {
  const size_t smem = static_cast<size_t>(N) * sizeof(float);
  return launch_select_any<true>(nullptr, parts, n_qc, B, G, N, k, force_last, idx, scores_out, smem, s, cu_in,
                                 cu_out, alive);
}

cudaError_t launch_flags_from_idx(const int32_t* idx, int B, int N, int k, uint8_t* flags,
                                  int* status, cudaStream_t s) {
  ZSAA_LAUNCH(flags_from_idx_kernel, dim3(B), dim3(256), 0, s, idx, N, k, flags, status);
  return cudaGetLastError();
}

cudaError_t launch_rows_norm(const void* src, const int32_t* tok, int vocab, int L,
                             const int32_t* idx, int N, int k, const int32_t* pos_in, int rows,
                             int d, const void* w, float eps, void* h_out, void* x_out,
                             int32_t* pos_out, int* status, cudaStream_t s, const int* cu_src,
                             const int* cu_dst, int nseq) {
  ZSAA_LAUNCH(rows_norm_bf16_kernel, dim3(row_blocks(rows)), dim3(32 * kWarpsPerBlock),
              static_cast<size_t>(d / 8) * 16, s,
              static_cast<const uint4*>(src), tok, vocab, L, idx, N, k, pos_in, rows, d / 8,
              static_cast<const uint4*>(w), eps, static_cast<uint4*>(h_out),
              static_cast<uint4*>(x_out), pos_out, status, cu_src, cu_dst, nseq);
  return cudaGetLastError();
}

cudaError_t launch_gather(const void* src, int B, int N, int k, int row_bytes, const int32_t* idx,
                          void* dst, const int32_t* pos_in, int32_t* pos_out, int* status,
                          cudaStream_t s) {
  const int total = B * k;
  ZSAA_LAUNCH(gather_rows_kernel<4>, dim3(row_blocks(total)), dim3(32 * kWarpsPerBlock), 0, s, 
      static_cast<const uint4*>(src), N, k, row_bytes / 16, idx, static_cast<uint4*>(dst),
      pos_in, pos_out, total, status);
  return cudaGetLastError();
}

cudaError_t launch_rope_f32(float* qkv, int rows, int ld, int rope_cols, int hd,
                            const int32_t* pos, const float* cos_t, const float* sin_t,
                            cudaStream_t s) {
  const int pairs = rope_cols / 2;
  dim3 grid((pairs + 127) / 128, rows);
  ZSAA_LAUNCH(rope_f32_kernel, dim3(grid), dim3(128), 0, s, qkv, rows, ld, rope_cols, hd, pos, cos_t, sin_t);
  return cudaGetLastError();
}

cudaError_t launch_cls_head(int dtype, const void* h, int B, int N, int d, const void* norm_w,
                            float eps, const void* W, int n_classes, float* out, cudaStream_t s,
                            const int* cu) {
  const size_t smem = static_cast<size_t>(d) * sizeof(float);
  if (dtype == ZSAA_BF16)
    ZSAA_LAUNCH(cls_head_kernel<bf16>, dim3(B), dim3(256), smem, s, static_cast<const bf16*>(h), N, d,
                                               static_cast<const bf16*>(norm_w), eps,
                                               static_cast<const bf16*>(W), n_classes, out, cu);
  else
    ZSAA_LAUNCH(cls_head_kernel<float>, dim3(B), dim3(256), smem, s, static_cast<const float*>(h), N, d,
                                                static_cast<const float*>(norm_w), eps,
                                                static_cast<const float*>(W), n_classes, out, cu);
  return cudaGetLastError();
}

}  // namespace zsaa
