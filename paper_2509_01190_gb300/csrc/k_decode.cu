// Generation over the pruned KV cache.
//
// Sec. 3.3 removes a pruned row from every later layer, so after a pruned
// prefill layer l holds the keys and values of only the rows it ran on.  A
// generated token attends, in layer l, to those rows plus the tokens generated
// before it and itself; generated tokens are never pruned.
//
// Cache of one layer: K and V bf16 [B, Hkv, cap, hd] (rows of one sequence and
// KV group contiguous, so a decode CTA streams them linearly), positions int32
// [B, cap].  The decode kernels read the step counter from device memory, so a
// captured decode step replays unchanged at every position.
#include "common.cuh"
#include "kernels.h"

namespace zsaa {
namespace {

__device__ __forceinline__ float bf16_round_f(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}

// One thread per 16-byte chunk; consecutive threads read consecutive chunks of
// a qkv row (key heads, then value heads).
__global__ void kv_write_kernel(const bf16* __restrict__ qkv, int ld,
                                const int32_t* __restrict__ pos, int B, int N, int Hq, int Hkv,
                                int hd, KvLayer c) {
  pdl_trigger();
  pdl_wait();
  const int cpr = hd / 8;
  const long long total = static_cast<long long>(B) * N * 2 * Hkv * cpr;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int ch = static_cast<int>(i % cpr);
    long long r = i / cpr;
    const int g = static_cast<int>(r % Hkv);
    r /= Hkv;
    const int kv = static_cast<int>(r % 2);
    r /= 2;
    const int j = static_cast<int>(r % N);
    const int b = static_cast<int>(r / N);
    const uint4* src = reinterpret_cast<const uint4*>(
                           qkv + (static_cast<size_t>(b) * N + j) * ld + static_cast<size_t>(Hq + kv * Hkv + g) * hd) +
                       ch;
    bf16* base = static_cast<bf16*>(kv ? c.v : c.k);
    uint4* dst = reinterpret_cast<uint4*>(
                     base + ((static_cast<size_t>(b) * Hkv + g) * c.cap + j) * static_cast<size_t>(hd)) +
                 ch;
    *dst = *src;
    if (g == 0 && kv == 0 && ch == 0)
      c.pos[static_cast<size_t>(b) * c.cap + j] = pos[static_cast<size_t>(b) * N + j];
  }
}

// One CTA per (KV group, sequence): RoPE and bf16 rounding of the group's PER
// query heads and of its key, append of key/value to the cache, then Eq. 1 of
// the PER queries over the cached rows.  8 warps take interleaved blocks of 32
// keys (one key per lane for the dot products, then one head dimension slice
// per lane for P V) with an online softmax in the log2 domain; the warps'
// partial results are merged at the end.
// W warps per CTA: the 32-key blocks are walked serially within a warp, so
// more warps shorten the chain (8: registers stay unspilled at 255 a thread).
template <int HD, int PER>
constexpr int decode_warps() { return 8; }

template <int HD, int PER>
__global__ void __launch_bounds__(decode_warps<HD, PER>() * 32)
    decode_attn_kernel(const float* __restrict__ qkv32, int ld, int Hq, int Hkv, KvLayer c,
                       const int* __restrict__ step, int L0, const float* __restrict__ cos_t,
                       const float* __restrict__ sin_t, bf16* __restrict__ out) {
  pdl_trigger();
  constexpr int HALF = HD / 2, DPL = HD / 32;  // head dims per lane in P V
  __shared__ __align__(16) float qs[PER][HD];
  constexpr int W = decode_warps<HD, PER>();
  __shared__ float wm[W][PER], wl[W][PER];
  __shared__ float wacc[W][PER][HD];
  const int g = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait();
  const int t = *step;
  const int p = L0 + t;
  const int row = c.base + t;
  const float* src = qkv32 + static_cast<size_t>(b) * ld;
  bf16* Kc = static_cast<bf16*>(c.k) + (static_cast<size_t>(b) * Hkv + g) * c.cap * static_cast<size_t>(HD);
  bf16* Vc = static_cast<bf16*>(c.v) + (static_cast<size_t>(b) * Hkv + g) * c.cap * static_cast<size_t>(HD);

  for (int i = threadIdx.x; i < (PER + 1) * HALF; i += blockDim.x) {
    const int h = i / HALF, dd = i % HALF;  // h < PER: query head g*PER + h; h == PER: key head g
    const float* x = src + static_cast<size_t>(h < PER ? g * PER + h : Hq + g) * HD;
    const float cs = cos_t[static_cast<size_t>(p) * HALF + dd];
    const float sn = sin_t[static_cast<size_t>(p) * HALF + dd];
    const float a = x[dd], bb = x[dd + HALF];
    const float y1 = a * cs - bb * sn, y2 = bb * cs + a * sn;
    if (h < PER) {
      qs[h][dd] = bf16_round_f(y1);
      qs[h][dd + HALF] = bf16_round_f(y2);
    } else {
      Kc[static_cast<size_t>(row) * HD + dd] = __float2bfloat16_rn(y1);
      Kc[static_cast<size_t>(row) * HD + dd + HALF] = __float2bfloat16_rn(y2);
    }
  }
  for (int dd = threadIdx.x; dd < HD; dd += blockDim.x)
    Vc[static_cast<size_t>(row) * HD + dd] =
        __float2bfloat16_rn(src[static_cast<size_t>(Hq + Hkv + g) * HD + dd]);
  if (g == 0 && threadIdx.x == 0) c.pos[static_cast<size_t>(b) * c.cap + row] = p;
  __syncthreads();  // the appended row is read below by other threads of this CTA

  const float scale = 1.4426950408889634f * rsqrtf(static_cast<float>(HD));  // log2(e)/sqrt(hd)
  const int n_keys = row + 1;
  float m[PER], l[PER], acc[PER][DPL];
#pragma unroll
  for (int h = 0; h < PER; ++h) {
    m[h] = -INFINITY;
    l[h] = 0.f;
#pragma unroll
    for (int e = 0; e < DPL; ++e) acc[h][e] = 0.f;
  }
  for (int j0 = warp * 32; j0 < n_keys; j0 += W * 32) {
    const int j = j0 + lane;
    const int nb = min(32, n_keys - j0);
    // this lane's head-dim slice of the block's 32 value rows, requested with
    // the key row below so that both memory latencies overlap
    uint32_t vw[32][DPL / 2];
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
      const bf16* vr = Vc + static_cast<size_t>(j0 + (jj < nb ? jj : 0)) * HD + lane * DPL;
      if constexpr (DPL == 2) {
        vw[jj][0] = *reinterpret_cast<const uint32_t*>(vr);
      } else {
        const uint2 w = *reinterpret_cast<const uint2*>(vr);
        vw[jj][0] = w.x;
        vw[jj][1] = w.y;
      }
    }
    float sc[PER];
    if (j < n_keys) {
      float dot[PER];
#pragma unroll
      for (int h = 0; h < PER; ++h) dot[h] = 0.f;
      const uint4* kr = reinterpret_cast<const uint4*>(Kc + static_cast<size_t>(j) * HD);
#pragma unroll
      for (int ch = 0; ch < HD / 8; ++ch) {
        const uint4 kv = kr[ch];
        const uint32_t w[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float k0 = __uint_as_float(w[e] << 16), k1 = __uint_as_float(w[e] & 0xffff0000u);
#pragma unroll
          for (int h = 0; h < PER; ++h)
            dot[h] = fmaf(qs[h][ch * 8 + 2 * e + 1], k1, fmaf(qs[h][ch * 8 + 2 * e], k0, dot[h]));
        }
      }
#pragma unroll
      for (int h = 0; h < PER; ++h) sc[h] = dot[h] * scale;
    } else {
#pragma unroll
      for (int h = 0; h < PER; ++h) sc[h] = -INFINITY;
    }
    float pj[PER];
#pragma unroll
    for (int h = 0; h < PER; ++h) {
      float mb = sc[h];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, o));
      const float mn = fmaxf(m[h], mb);  // finite: lane 0's key exists
      const float corr = exp2f(m[h] - mn);
      pj[h] = exp2f(sc[h] - mn);
      float ps = pj[h];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
      l[h] = l[h] * corr + ps;
#pragma unroll
      for (int e = 0; e < DPL; ++e) acc[h][e] *= corr;
      m[h] = mn;
    }
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
      if (jj < nb) {  // warp-uniform
        float vv[DPL];
#pragma unroll
        for (int e2 = 0; e2 < DPL / 2; ++e2) {
          vv[2 * e2] = __uint_as_float(vw[jj][e2] << 16);
          vv[2 * e2 + 1] = __uint_as_float(vw[jj][e2] & 0xffff0000u);
        }
#pragma unroll
        for (int h = 0; h < PER; ++h) {
          const float pk = __shfl_sync(0xffffffffu, pj[h], jj);
#pragma unroll
          for (int e = 0; e < DPL; ++e) acc[h][e] = fmaf(pk, vv[e], acc[h][e]);
        }
      }
    }
  }
  if (lane == 0) {
#pragma unroll
    for (int h = 0; h < PER; ++h) {
      wm[warp][h] = m[h];
      wl[warp][h] = l[h];
    }
  }
#pragma unroll
  for (int h = 0; h < PER; ++h)
#pragma unroll
    for (int e = 0; e < DPL; ++e) wacc[warp][h][lane * DPL + e] = acc[h][e];
  __syncthreads();
  for (int i = threadIdx.x; i < PER * HD; i += blockDim.x) {
    const int h = i / HD, dd = i % HD;
    float mx = -INFINITY;
#pragma unroll
    for (int w = 0; w < W; ++w) mx = fmaxf(mx, wm[w][h]);
    float num = 0.f, den = 0.f;
#pragma unroll
    for (int w = 0; w < W; ++w) {
      const float f = wm[w][h] == -INFINITY ? 0.f : exp2f(wm[w][h] - mx);
      num = fmaf(f, wacc[w][h][dd], num);
      den = fmaf(f, wl[w][h], den);
    }
    out[static_cast<size_t>(b) * Hq * HD + static_cast<size_t>(g * PER + h) * HD + dd] =
        __float2bfloat16_rn(num / den);
  }
}

__global__ void advance_kernel(int* step) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) *step += 1;
}

template <int HD>
cudaError_t run_decode(int per, dim3 grid, cudaStream_t s, const float* qkv32, int ld, int Hq,
                       int Hkv, const KvLayer& c, const int* step, int L0, const float* cos_t,
                       const float* sin_t, bf16* out) {
  switch (per) {
    case 1: ZSAA_LAUNCH(decode_attn_kernel<HD, 1>, grid, dim3(decode_warps<HD, 1>() * 32), 0, s, qkv32, ld, Hq, Hkv, c, step, L0, cos_t, sin_t, out); break;
    case 2: ZSAA_LAUNCH(decode_attn_kernel<HD, 2>, grid, dim3(decode_warps<HD, 2>() * 32), 0, s, qkv32, ld, Hq, Hkv, c, step, L0, cos_t, sin_t, out); break;
    case 4: ZSAA_LAUNCH(decode_attn_kernel<HD, 4>, grid, dim3(decode_warps<HD, 4>() * 32), 0, s, qkv32, ld, Hq, Hkv, c, step, L0, cos_t, sin_t, out); break;
    case 8: ZSAA_LAUNCH(decode_attn_kernel<HD, 8>, grid, dim3(decode_warps<HD, 8>() * 32), 0, s, qkv32, ld, Hq, Hkv, c, step, L0, cos_t, sin_t, out); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_kv_write(const void* qkv, int ld, const int32_t* pos, int B, int N, int Hq,
                            int Hkv, int hd, const KvLayer& c, cudaStream_t s) {
  const long long total = static_cast<long long>(B) * N * 2 * Hkv * (hd / 8);
  const long long want = (total + 255) / 256;
  const int grid = static_cast<int>(want < 4096 ? (want > 0 ? want : 1) : 4096);
  ZSAA_LAUNCH(kv_write_kernel, dim3(grid), dim3(256), 0, s, static_cast<const bf16*>(qkv), ld, pos,
              B, N, Hq, Hkv, hd, c);
  return cudaSuccess;
}

cudaError_t launch_decode_attention(const float* qkv32, int ld, int B, int Hq, int Hkv, int hd,
                                    const KvLayer& c, const int* step, int L0, const float* cos_t,
                                    const float* sin_t, void* out, cudaStream_t s) {
  const int per = Hq / Hkv;
  const dim3 grid(Hkv, B);
  bf16* o = static_cast<bf16*>(out);
  if (hd == 64) return run_decode<64>(per, grid, s, qkv32, ld, Hq, Hkv, c, step, L0, cos_t, sin_t, o);
  if (hd == 128) return run_decode<128>(per, grid, s, qkv32, ld, Hq, Hkv, c, step, L0, cos_t, sin_t, o);
  return cudaErrorInvalidValue;
}

cudaError_t launch_decode_advance(int* step, cudaStream_t s) {
  ZSAA_LAUNCH(advance_kernel, dim3(1), dim3(32), 0, s, step);
  return cudaSuccess;
}

}  // namespace zsaa
