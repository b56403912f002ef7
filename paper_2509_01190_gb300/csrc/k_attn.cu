// Causal grouped-query attention (Eq. 1) and the soft-score column mass
// (Sec. 3.2: soft-score times V gives each V row's contribution).
//
// qkv is the packed projection [B*N, (Hq + 2 Hkv) hd]: per row Hq query heads
// (RoPE applied), Hkv key heads (RoPE applied), Hkv value heads.  Query head h
// reads KV head h / (Hq / Hkv).
//
// attention: out[b*N+i, h*hd:] = sum_j P[i,j] v_j with P = softmax over j <= i of
//   q_i.k_j / sqrt(hd); lse2[b,h,i] = log2 of the normaliser of the logits
//   scaled by log2(e)/sqrt(hd) (so P[i,j] = exp2(s_ij * c - lse2[i])).
// column mass: C[b,g,j] = sum over heads h of group g, queries i >= j, of
//   P[i,j], recomputed from q, k and lse2 (no N x N matrix is stored).
//
// bf16 path: FlashAttention-style tiles on mma.sync m16n8k16 (64 queries x 64
// keys per step, 4 warps x 16 rows), online softmax in fp32; the probabilities
// enter P V as a hi/lo pair of bf16 matrices.  The column-mass
// pass sweeps key blocks outer / query blocks inner so each CTA owns its
// columns and sums them in registers (deterministic, no atomics).
// fp32 path: plain CUDA-core kernels (one warp per row / column).
#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

// byte offset of 16-byte chunk c of row r in a tile with ROWB bytes per row,
// chunks XOR-swizzled by the row's low 3 bits (conflict-free ldmatrix)
template <int ROWB>
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>(r * ROWB + ((c ^ (r & 7)) << 4));
}

// cp.async a [64 x HD] bf16 tile whose rows start at g + (row0 + r) * ld; rows
// at or beyond n_valid are zero-filled.
template <int HD>
__device__ __forceinline__ void load_tile64(uint32_t sbase, const bf16* g, size_t ld, int row0,
                                            int n_valid) {
  constexpr int CH = HD / 8;
  for (int i = threadIdx.x; i < 64 * CH; i += 128) {
    const int r = i / CH, c = i % CH;
    const bool v = row0 + r < n_valid;
    const bf16* src = g + (v ? static_cast<size_t>(row0 + r) * ld : 0) + c * 8;
    cp_async16(sbase + swz<HD * 2>(r, c), src, v);
  }
}

template <int HD>
__global__ void __launch_bounds__(128)
    attn_fwd_bf16_kernel(const bf16* __restrict__ qkv, int Ns, int Hq, int Hkv,
                         bf16* __restrict__ out, float* __restrict__ lse2, float scale_log2,
                         int causal, const int* __restrict__ cu,
                         const uint8_t* __restrict__ key_alive) {
  pdl_trigger();
  pdl_wait();
  constexpr int ROWB = HD * 2;
  constexpr int TILE = 64 * ROWB;
  extern __shared__ __align__(128) uint8_t sm[];
  const uint32_t sQ = smem_u32(sm);
  const uint32_t sK0 = sQ + TILE, sV0 = sQ + 3 * TILE;  // K: 2 buffers, V: 2 buffers

  const int qb = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  // fixed length: N = Ns rows per sequence; packed variable length: this
  // sequence's rows [cu[b], cu[b+1]) (Ns = the longest: grid and lse stride)
  const size_t row0 = cu ? static_cast<size_t>(cu[b]) : static_cast<size_t>(b) * Ns;
  const int N = cu ? cu[b + 1] - cu[b] : Ns;
  if (qb * 64 >= N) return;
  // masked mode (Appendix B): keys whose flag is 0 are hidden from every query
  const uint8_t* ka = key_alive ? key_alive + static_cast<size_t>(b) * Ns : nullptr;
  const int g = h / (Hq / Hkv);
  const size_t ld = static_cast<size_t>(Hq + 2 * Hkv) * HD;
  const bf16* base = qkv + row0 * ld;
  const bf16* Qg = base + h * HD;
  const bf16* Kg = base + (Hq + g) * HD;
  const bf16* Vg = base + (Hq + Hkv + g) * HD;
  const int q0 = qb * 64;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;

  const int kv_end = causal ? min(N, q0 + 64) : N;
  const int n_kb = (kv_end + 63) / 64;

  load_tile64<HD>(sQ, Qg, ld, q0, N);
  load_tile64<HD>(sK0, Kg, ld, 0, N);
  load_tile64<HD>(sV0, Vg, ld, 0, N);
  cp_async_commit();

  uint32_t qf[HD / 16][4];
  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_lo = -INFINITY, m_hi = -INFINITY, l_lo = 0.f, l_hi = 0.f;
  const int i_lo = q0 + warp * 16 + gid, i_hi = i_lo + 8;

  for (int kb = 0; kb < n_kb; ++kb) {
    const int buf = kb & 1;
    if (kb + 1 < n_kb) {
      load_tile64<HD>(sK0 + (buf ^ 1) * TILE, Kg, ld, (kb + 1) * 64, N);
      load_tile64<HD>(sV0 + (buf ^ 1) * TILE, Vg, ld, (kb + 1) * 64, N);
    }
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (kb == 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int mi = lane >> 3;
        const int r = warp * 16 + (mi & 1) * 8 + (lane & 7);
        ldsm_x4(sQ + swz<ROWB>(r, kk * 2 + (mi >> 1)), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    const uint32_t sK = sK0 + buf * TILE, sV = sV0 + buf * TILE;
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int mi = lane >> 3;
        const int r = np * 16 + (mi >> 1) * 8 + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sK + swz<ROWB>(r, kk * 2 + (mi & 1)), b0, b1, b2, b3);
        mma_bf16_16816(s[2 * np], qf[kk], b0, b1);
        mma_bf16_16816(s[2 * np + 1], qf[kk], b2, b3);
      }
    }
    // scale, causal / length mask, online softmax
    const int k0 = kb * 64;
    float mx_lo = -INFINITY, mx_hi = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = k0 + nt * 8 + 2 * tig + e;
        float a = s[nt][e] * scale_log2, c = s[nt][2 + e] * scale_log2;
        const bool dead = j >= N || (ka != nullptr && ka[j] == 0);
        if ((causal && j > i_lo) || dead) a = -INFINITY;
        if ((causal && j > i_hi) || dead) c = -INFINITY;
        s[nt][e] = a;
        s[nt][2 + e] = c;
        mx_lo = fmaxf(mx_lo, a);
        mx_hi = fmaxf(mx_hi, c);
      }
    }
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 1));
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 2));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 1));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 2));
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
    const float base_lo = mn_lo == -INFINITY ? 0.f : mn_lo;
    const float base_hi = mn_hi == -INFINITY ? 0.f : mn_hi;
    const float al_lo = exp2f(m_lo - base_lo), al_hi = exp2f(m_hi - base_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    l_lo *= al_lo;
    l_hi *= al_hi;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      o[i][0] *= al_lo;
      o[i][1] *= al_lo;
      o[i][2] *= al_hi;
      o[i][3] *= al_hi;
    }
    // P as a pair of bf16 matrices, P = P_hi + P_lo, so P V keeps ~16 bits of P
    // (one bf16 P would cost ~0.1% relative error in every output).
    uint32_t ph[4][4], pl[4][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = exp2f(s[nt][0] - base_lo), p1 = exp2f(s[nt][1] - base_lo);
      const float p2 = exp2f(s[nt][2] - base_hi), p3 = exp2f(s[nt][3] - base_hi);
      l_lo += p0 + p1;
      l_hi += p2 + p3;
      const uint32_t h01 = pack_bf16x2(p0, p1), h23 = pack_bf16x2(p2, p3);
      ph[nt >> 1][(nt & 1) * 2 + 0] = h01;
      ph[nt >> 1][(nt & 1) * 2 + 1] = h23;
      pl[nt >> 1][(nt & 1) * 2 + 0] = pack_bf16x2(p0 - bf16lo(h01), p1 - bf16hi(h01));
      pl[nt >> 1][(nt & 1) * 2 + 1] = pack_bf16x2(p2 - bf16lo(h23), p3 - bf16hi(h23));
    }
    // O += P_hi V + P_lo V
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        const int mi = lane >> 3;
        const int r = j * 16 + (mi & 1) * 8 + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sV + swz<ROWB>(r, dp * 2 + (mi >> 1)), b0, b1, b2, b3);
        mma_bf16_16816(o[2 * dp], ph[j], b0, b1);
        mma_bf16_16816(o[2 * dp + 1], ph[j], b2, b3);
        mma_bf16_16816(o[2 * dp], pl[j], b0, b1);
        mma_bf16_16816(o[2 * dp + 1], pl[j], b2, b3);
      }
    }
    __syncthreads();
  }
  cp_async_wait<0>();
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 1);
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 2);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 1);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 2);
  const float inv_lo = l_lo > 0.f ? 1.f / l_lo : 0.f, inv_hi = l_hi > 0.f ? 1.f / l_hi : 0.f;
  const size_t ldo = static_cast<size_t>(Hq) * HD;
  if (i_lo < N) {
    bf16* orow = out + (row0 + i_lo) * ldo + h * HD;
#pragma unroll
    for (int nt = 0; nt < HD / 8; ++nt)
      *reinterpret_cast<uint32_t*>(orow + nt * 8 + 2 * tig) =
          pack_bf16x2(o[nt][0] * inv_lo, o[nt][1] * inv_lo);
    if (tig == 0) lse2[(static_cast<size_t>(b) * Hq + h) * Ns + i_lo] = m_lo + log2f(l_lo);
  }
  if (i_hi < N) {
    bf16* orow = out + (row0 + i_hi) * ldo + h * HD;
#pragma unroll
    for (int nt = 0; nt < HD / 8; ++nt)
      *reinterpret_cast<uint32_t*>(orow + nt * 8 + 2 * tig) =
          pack_bf16x2(o[nt][2] * inv_hi, o[nt][3] * inv_hi);
    if (tig == 0) lse2[(static_cast<size_t>(b) * Hq + h) * Ns + i_hi] = m_hi + log2f(l_hi);
  }
}

// Column mass: CTA (key block kb, query chunk qc, KV head g * B + b).  Warp w
// owns keys kb*64 + w*16 .. +16 as the A operand; the query tiles of chunk qc
// (q_per blocks of 64, only those at or after the key block) are the B
// operand, for every query head of group g.  The CTA writes its partial column
// sums, times ||v_j|| of group g when weight_vnorm is set (the score of R1 is
// linear in the column mass), to parts[qc][b][g][j]; a reduce kernel sums
// the chunks in a fixed order.
template <int HD>
__global__ void __launch_bounds__(128)
    colmass_bf16_kernel(const bf16* __restrict__ qkv, const float* __restrict__ lse2, int N,
                        int Hq, int Hkv, int B, int q_per, int weight_vnorm,
                        float* __restrict__ parts, float scale_log2, int causal) {
  pdl_trigger();
  pdl_wait();
  constexpr int ROWB = HD * 2;
  constexpr int TILE = 64 * ROWB;
  extern __shared__ __align__(128) uint8_t sm[];
  float* sL = reinterpret_cast<float*>(sm + 3 * TILE);  // 2 x 64 lse values
  const uint32_t sK = smem_u32(sm), sQ0 = sK + TILE;

  const int kb = blockIdx.x, qc = blockIdx.y;
  const int g = blockIdx.z % Hkv, b = blockIdx.z / Hkv;
  const int per = Hq / Hkv;
  const size_t ld = static_cast<size_t>(Hq + 2 * Hkv) * HD;
  const bf16* base = qkv + static_cast<size_t>(b) * N * ld;
  const bf16* Kg = base + (Hq + g) * HD;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;
  const int j_lo = kb * 64 + warp * 16 + gid, j_hi = j_lo + 8;
  const int n_qb = (N + 63) / 64;
  const int qb0 = max(causal ? kb : 0, qc * q_per), qb1 = min(n_qb, (qc + 1) * q_per);
  const int nq = qb1 > qb0 ? qb1 - qb0 : 0;
  const int steps = per * nq;

  auto issue = [&](int step, int buf) {
    const int hh = step / nq, qb = qb0 + step % nq;
    const int h = g * per + hh;
    load_tile64<HD>(sQ0 + buf * TILE, base + h * HD, ld, qb * 64, N);
    for (int i = threadIdx.x; i < 64; i += 128) {
      const int q = qb * 64 + i;
      sL[buf * 64 + i] = q < N ? lse2[(static_cast<size_t>(b) * Hq + h) * N + q] : 0.f;
    }
  };

  float acc_lo = 0.f, acc_hi = 0.f;
  if (steps > 0) {
    load_tile64<HD>(sK, Kg, ld, kb * 64, N);
    issue(0, 0);
    cp_async_commit();
    uint32_t kf[HD / 16][4];
    for (int step = 0; step < steps; ++step) {
      const int buf = step & 1;
      if (step + 1 < steps) issue(step + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
      __syncthreads();
      if (step == 0) {
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const int mi = lane >> 3;
          const int r = warp * 16 + (mi & 1) * 8 + (lane & 7);
          ldsm_x4(sK + swz<ROWB>(r, kk * 2 + (mi >> 1)), kf[kk][0], kf[kk][1], kf[kk][2], kf[kk][3]);
        }
      }
      const int qb = qb0 + step % nq;
      const uint32_t sQ = sQ0 + buf * TILE;
      float sacc[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) sacc[nt][0] = sacc[nt][1] = sacc[nt][2] = sacc[nt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int mi = lane >> 3;
          const int r = np * 16 + (mi >> 1) * 8 + (lane & 7);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(sQ + swz<ROWB>(r, kk * 2 + (mi & 1)), b0, b1, b2, b3);
          mma_bf16_16816(sacc[2 * np], kf[kk], b0, b1);
          mma_bf16_16816(sacc[2 * np + 1], kf[kk], b2, b3);
        }
      }
      const float* Lq = sL + buf * 64;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int qi = nt * 8 + 2 * tig + e;
          const int i = qb * 64 + qi;
          if (i < N) {
            const float l = Lq[qi];
            if (!causal || i >= j_lo) acc_lo += exp2f(sacc[nt][e] * scale_log2 - l);
            if (!causal || i >= j_hi) acc_hi += exp2f(sacc[nt][2 + e] * scale_log2 - l);
          }
        }
      }
      __syncthreads();
    }
    cp_async_wait<0>();
  }
  acc_lo += __shfl_xor_sync(0xffffffffu, acc_lo, 1);
  acc_lo += __shfl_xor_sync(0xffffffffu, acc_lo, 2);
  acc_hi += __shfl_xor_sync(0xffffffffu, acc_hi, 1);
  acc_hi += __shfl_xor_sync(0xffffffffu, acc_hi, 2);
  if (weight_vnorm) {
    // ||v_j|| of group g: the quad (tig = 0..3) splits the hd dims of rows j_lo, j_hi
    const bf16* Vg = base + (Hq + Hkv + g) * HD;
    float ss_lo = 0.f, ss_hi = 0.f;
    constexpr int QD = HD / 4;
    if (j_lo < N) {
      const uint4* v = reinterpret_cast<const uint4*>(Vg + static_cast<size_t>(j_lo) * ld + tig * QD);
#pragma unroll
      for (int q = 0; q < QD / 8; ++q) {
        const uint4 u = v[q];
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) ss_lo += bf16lo(w[e]) * bf16lo(w[e]) + bf16hi(w[e]) * bf16hi(w[e]);
      }
    }
    if (j_hi < N) {
      const uint4* v = reinterpret_cast<const uint4*>(Vg + static_cast<size_t>(j_hi) * ld + tig * QD);
#pragma unroll
      for (int q = 0; q < QD / 8; ++q) {
        const uint4 u = v[q];
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) ss_hi += bf16lo(w[e]) * bf16lo(w[e]) + bf16hi(w[e]) * bf16hi(w[e]);
      }
    }
    ss_lo += __shfl_xor_sync(0xffffffffu, ss_lo, 1);
    ss_lo += __shfl_xor_sync(0xffffffffu, ss_lo, 2);
    ss_hi += __shfl_xor_sync(0xffffffffu, ss_hi, 1);
    ss_hi += __shfl_xor_sync(0xffffffffu, ss_hi, 2);
    acc_lo *= sqrtf(ss_lo);
    acc_hi *= sqrtf(ss_hi);
  }
  if (tig == 0) {
    float* P = parts + ((static_cast<size_t>(qc) * B + b) * Hkv + g) * N;
    if (j_lo < N) P[j_lo] = acc_lo;
    if (j_hi < N) P[j_hi] = acc_hi;
  }
}

// out[b][g][j] = sum_qc parts[qc][b][g][j]                      (sum_groups = 0)
// out[b][j]    = sum_qc sum_g parts[qc][b][g][j]                 (sum_groups = 1)
__global__ void colmass_reduce_kernel(const float* __restrict__ parts, int n_qc, int B, int G,
                                      int N, int sum_groups, float* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int total = sum_groups ? B * N : B * G * N;
  if (idx >= total) return;
  const size_t plane = static_cast<size_t>(B) * G * N;
  float acc = 0.f;
  if (sum_groups) {
    const int b = idx / N, j = idx % N;
    for (int qc = 0; qc < n_qc; ++qc)
      for (int g = 0; g < G; ++g) acc += parts[qc * plane + (static_cast<size_t>(b) * G + g) * N + j];
  } else {
    for (int qc = 0; qc < n_qc; ++qc) acc += parts[qc * plane + idx];
  }
  out[idx] = acc;
}

// fp32 attention: one warp per (query i, head h, batch b).
__global__ void attn_fwd_f32_kernel(const float* __restrict__ qkv, int N, int Hq, int Hkv, int hd,
                                    float* __restrict__ out, float* __restrict__ lse2,
                                    float scale_log2, int causal) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int h = blockIdx.y, b = blockIdx.z, lane = threadIdx.x & 31;
  if (i >= N) return;
  const int g = h / (Hq / Hkv);
  const size_t ld = static_cast<size_t>(Hq + 2 * Hkv) * hd;
  const float* base = qkv + static_cast<size_t>(b) * N * ld;
  const float* q = base + i * ld + h * hd;
  const int jend = causal ? i + 1 : N;  // keys [0, jend)
  // pass 1: max and normaliser (per lane over its keys, then merged)
  float m = -INFINITY, l = 0.f;
  for (int j = lane; j < jend; j += 32) {
    const float* k = base + j * ld + (Hq + g) * hd;
    float s = 0.f;
    for (int e = 0; e < hd; ++e) s = fmaf(q[e], k[e], s);
    s *= scale_log2;
    const float mn = fmaxf(m, s);
    l = l * exp2f(m - mn) + exp2f(s - mn);
    m = mn;
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), l2 = __shfl_xor_sync(0xffffffffu, l, o);
    const float mn = fmaxf(m, m2);
    const float bm = mn == -INFINITY ? 0.f : mn;
    l = l * exp2f(m - bm) + l2 * exp2f(m2 - bm);
    m = mn;
  }
  const float lse = m + log2f(l);
  // pass 2: output, each lane owns dims lane, lane+32, ...
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int j0 = 0; j0 < jend; j0 += 32) {
    const int j = j0 + lane;
    float p = 0.f;
    if (j < jend) {
      const float* k = base + j * ld + (Hq + g) * hd;
      float s = 0.f;
      for (int e = 0; e < hd; ++e) s = fmaf(q[e], k[e], s);
      p = exp2f(s * scale_log2 - lse);
    }
    const int cnt = min(32, jend - j0);
    for (int t = 0; t < cnt; ++t) {
      const float pt = __shfl_sync(0xffffffffu, p, t);
      const float* v = base + (j0 + t) * ld + (Hq + Hkv + g) * hd;
      for (int e = lane, c = 0; e < hd; e += 32, ++c) acc[c] = fmaf(pt, v[e], acc[c]);
    }
  }
  float* orow = out + (static_cast<size_t>(b) * N + i) * Hq * hd + h * hd;
  for (int e = lane, c = 0; e < hd; e += 32, ++c) orow[e] = acc[c];
  if (lane == 0) lse2[(static_cast<size_t>(b) * Hq + h) * N + i] = lse;
}

// fp32 column mass: one warp per (key j, KV head g, batch b); one query chunk.
__global__ void colmass_f32_kernel(const float* __restrict__ qkv, const float* __restrict__ lse2,
                                   int N, int Hq, int Hkv, int hd, int B, int weight_vnorm,
                                   float* __restrict__ parts, float scale_log2, int causal) {
  pdl_trigger();
  pdl_wait();
  const int j = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int g = blockIdx.y, b = blockIdx.z, lane = threadIdx.x & 31;
  if (j >= N) return;
  const int per = Hq / Hkv;
  const size_t ld = static_cast<size_t>(Hq + 2 * Hkv) * hd;
  const float* base = qkv + static_cast<size_t>(b) * N * ld;
  const float* k = base + j * ld + (Hq + g) * hd;
  float acc = 0.f;
  for (int hh = 0; hh < per; ++hh) {
    const int h = g * per + hh;
    for (int i = (causal ? j : 0) + lane; i < N; i += 32) {
      const float* q = base + i * ld + h * hd;
      float s = 0.f;
      for (int e = 0; e < hd; ++e) s = fmaf(q[e], k[e], s);
      acc += exp2f(s * scale_log2 - lse2[(static_cast<size_t>(b) * Hq + h) * N + i]);
    }
  }
  acc = warp_sum(acc);
  if (weight_vnorm) {
    const float* v = base + j * ld + (Hq + Hkv + g) * hd;
    float ss = 0.f;
    for (int e = lane; e < hd; e += 32) ss = fmaf(v[e], v[e], ss);
    acc *= sqrtf(warp_sum(ss));
  }
  if (lane == 0) parts[(static_cast<size_t>(b) * Hkv + g) * N + j] = acc;
}

}  // namespace

cudaError_t launch_attention(int dtype, const void* qkv, int B, int N, int Hq, int Hkv, int hd,
                             void* out, float* lse, int causal, cudaStream_t s, const int* cu,
                             const uint8_t* key_alive) {
  if ((cu != nullptr || key_alive != nullptr) && dtype != ZSAA_BF16) return cudaErrorInvalidValue;
  const float scale_log2 = kLog2e / sqrtf(static_cast<float>(hd));
  if (dtype == ZSAA_F32) {
    dim3 grid((N + 3) / 4, Hq, B);
    ZSAA_LAUNCH(attn_fwd_f32_kernel, dim3(grid), dim3(128), 0, s, static_cast<const float*>(qkv), N, Hq, Hkv, hd,
                                             static_cast<float*>(out), lse, scale_log2, causal);
    return cudaGetLastError();
  }
  dim3 grid((N + 63) / 64, Hq, B);
  if (hd == 64) {
    const int smem = 5 * 64 * 128;
    static OncePerDevice once;
    const cudaError_t e = set_smem_limit_once(once, attn_fwd_bf16_kernel<64>, smem);
    if (e != cudaSuccess) return e;
    ZSAA_LAUNCH(attn_fwd_bf16_kernel<64>, dim3(grid), dim3(128), smem, s, static_cast<const bf16*>(qkv), N, Hq, Hkv,
                                                      static_cast<bf16*>(out), lse, scale_log2, causal, cu, key_alive);
  } else if (hd == 128) {
    const int smem = 5 * 64 * 256;
    static OncePerDevice once;
    const cudaError_t e = set_smem_limit_once(once, attn_fwd_bf16_kernel<128>, smem);
    if (e != cudaSuccess) return e;
    ZSAA_LAUNCH(attn_fwd_bf16_kernel<128>, dim3(grid), dim3(128), smem, s, static_cast<const bf16*>(qkv), N, Hq, Hkv,
                                                       static_cast<bf16*>(out), lse, scale_log2, causal, cu, key_alive);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

int colmass_chunks(int N) {
  const int n_qb = (N + 63) / 64;
  return (n_qb + kColmassQPer - 1) / kColmassQPer;
}

size_t colmass_parts_elems(int B, int N, int Hq, int Hkv) {
  const int tc_chunks = 2 * (Hq / Hkv);  // the tensor-core kernel: (head, column half)
  const int c = colmass_chunks(N) > tc_chunks ? colmass_chunks(N) : tc_chunks;
  return static_cast<size_t>(c) * B * Hkv * N;
}

namespace {
cudaError_t colmass_parts(int dtype, const void* qkv, const float* lse, const float* vnorm, int B,
                          int N, int Hq, int Hkv, int hd, int weight_vnorm, float* parts, int* n_qc,
                          int* status, int causal, cudaStream_t s, const int* cu = nullptr,
                          int rows = 0, const uint8_t* q_alive = nullptr) {
  // tensor-core path (with precomputed norms when they are needed)
  if (dtype == ZSAA_BF16 && status != nullptr && (!weight_vnorm || vnorm != nullptr))
    return launch_colmass_tc(qkv, lse, weight_vnorm ? vnorm : nullptr, B, N, Hq, Hkv, hd, parts,
                             status, n_qc, causal, s, cu, rows, q_alive);
  if (cu != nullptr || q_alive != nullptr) return cudaErrorInvalidValue;  // tensor-core path only
  const float scale_log2 = kLog2e / sqrtf(static_cast<float>(hd));
  if (dtype == ZSAA_F32) {
    *n_qc = 1;
    dim3 grid((N + 3) / 4, Hkv, B);
    ZSAA_LAUNCH(colmass_f32_kernel, dim3(grid), dim3(128), 0, s, static_cast<const float*>(qkv), lse, N, Hq, Hkv, hd, B,
                                            weight_vnorm, parts, scale_log2, causal);
    return cudaGetLastError();
  }
  *n_qc = colmass_chunks(N);
  dim3 grid((N + 63) / 64, *n_qc, Hkv * B);
  if (hd == 64) {
    const int smem = 3 * 64 * 128 + 2 * 64 * 4;
    static OncePerDevice once;
    const cudaError_t e = set_smem_limit_once(once, colmass_bf16_kernel<64>, smem);
    if (e != cudaSuccess) return e;
    ZSAA_LAUNCH(colmass_bf16_kernel<64>, dim3(grid), dim3(128), smem, s, static_cast<const bf16*>(qkv), lse, N, Hq,
                                                     Hkv, B, kColmassQPer, weight_vnorm, parts,
                                                     scale_log2, causal);
  } else if (hd == 128) {
    const int smem = 3 * 64 * 256 + 2 * 64 * 4;
    static OncePerDevice once;
    const cudaError_t e = set_smem_limit_once(once, colmass_bf16_kernel<128>, smem);
    if (e != cudaSuccess) return e;
    ZSAA_LAUNCH(colmass_bf16_kernel<128>, dim3(grid), dim3(128), smem, s, static_cast<const bf16*>(qkv), lse, N, Hq,
                                                      Hkv, B, kColmassQPer, weight_vnorm, parts,
                                                      scale_log2, causal);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_colmass(int dtype, const void* qkv, const float* lse, int B, int N, int Hq,
                           int Hkv, int hd, float* parts, float* C, int* status, int causal,
                           cudaStream_t s) {
  int n_qc = 1;
  cudaError_t e = colmass_parts(dtype, qkv, lse, nullptr, B, N, Hq, Hkv, hd, 0, parts, &n_qc, status,
                                causal, s);
  if (e != cudaSuccess) return e;
  const int total = B * Hkv * N;
  ZSAA_LAUNCH(colmass_reduce_kernel, dim3((total + 255) / 256), dim3(256), 0, s, parts, n_qc, B, Hkv, N, 0, C);
  return cudaGetLastError();
}

cudaError_t launch_position_parts(int dtype, const void* qkv, const float* lse, const float* vnorm,
                                  int B, int N, int Hq, int Hkv, int hd, int mode, float* parts,
                                  int* n_qc, int* status, int causal, cudaStream_t s, const int* cu,
                                  int rows, const uint8_t* q_alive) {
  return colmass_parts(dtype, qkv, lse, vnorm, B, N, Hq, Hkv, hd,
                       mode == ZSAA_SCORE_SOFTSCORE_VNORM ? 1 : 0, parts, n_qc, status, causal, s,
                       cu, rows, q_alive);
}

cudaError_t launch_position_scores(int dtype, const void* qkv, const float* lse, const float* vnorm,
                                   int B, int N, int Hq, int Hkv, int hd, int mode, float* parts,
                                   float* scores, int* status, int causal, cudaStream_t s) {
  int n_qc = 1;
  cudaError_t e = colmass_parts(dtype, qkv, lse, vnorm, B, N, Hq, Hkv, hd,
                                mode == ZSAA_SCORE_SOFTSCORE_VNORM ? 1 : 0, parts, &n_qc, status,
                                causal, s);
  if (e != cudaSuccess) return e;
  const int total = B * N;
  ZSAA_LAUNCH(colmass_reduce_kernel, dim3((total + 255) / 256), dim3(256), 0, s, parts, n_qc, B, Hkv, N, 1, scores);
  return cudaGetLastError();
}

}  // namespace zsaa
