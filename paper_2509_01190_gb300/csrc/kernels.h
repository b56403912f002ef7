// Host-side launchers of the library's kernels (internal; not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace zsaa {

// ---- row kernels (k_rows.cu)
cudaError_t launch_embed(int dtype, const void* E, const int32_t* tok, int rows, int L, int vocab,
                         int d, void* h, int32_t* pos, int* status, cudaStream_t s);
cudaError_t launch_rmsnorm(int dtype, const void* h, const void* w, int rows, int d, float eps,
                           void* x, cudaStream_t s);
cudaError_t launch_row_norm(int dtype, const void* h, int rows, int d, float* scores,
                            cudaStream_t s);
cudaError_t launch_select(const float* scores, int B, int N, int k, int force_last, int32_t* idx,
                          cudaStream_t s);
// Top-k from column-mass partials parts[n_qc][B][G][N] (scores summed in shared
// memory, copied to scores_out when not null); N <= kSelectPartsMaxN.
constexpr int kSelectPartsMaxN = 12288;
// Variable length (cu_in / cu_out: packed row offsets [B+1] before / after the
// selection): sequence b has cu_in[b+1]-cu_in[b] candidates, keeps
// cu_out[b+1]-cu_out[b], partials at stride N (the longest), idx and scores
// written packed at cu_out[b] / cu_in[b].
cudaError_t launch_select_parts(const float* parts, int n_qc, int B, int G, int N, int k,
                                int force_last, int32_t* idx, float* scores_out, cudaStream_t s,
                                const int* cu_in = nullptr, const int* cu_out = nullptr,
                                uint8_t* alive = nullptr);
// alive (masked mode, fixed length): [B, N] flags; only flagged rows compete
// (k includes the forced last row), and afterwards exactly the kept rows are
// flagged.  idx then holds positions 0..N-1.
// bf16 rows: h_out[r] = source row, x_out[r] = RMSNorm(h_out[r]) * w, pos_out[r].
// Embedding when idx == nullptr (rows = B*L, source row tok[r] of E);
// otherwise compaction (rows = B*k, source row b*N + idx[r] of h).
// d % 8 == 0 and d <= kRowsNormMaxD.
constexpr int kRowsNormMaxD = 8 * 32 * 16;
// Variable length: cu_dst (offsets of the written rows; nseq sequences) gives
// the sequence of a row and, for the embedding, pos = r - cu_dst[b]; cu_src
// (offsets of the source rows) places compaction index j at row cu_src[b] + j.
cudaError_t launch_rows_norm(const void* src, const int32_t* tok, int vocab, int L,
                             const int32_t* idx, int N, int k, const int32_t* pos_in, int rows,
                             int d, const void* w, float eps, void* h_out, void* x_out,
                             int32_t* pos_out, int* status, cudaStream_t s,
                             const int* cu_src = nullptr, const int* cu_dst = nullptr,
                             int nseq = 0);
// flags[b, :N] = 0 except 1 at positions idx[b, :k] (masked mode, forced choice).
cudaError_t launch_flags_from_idx(const int32_t* idx, int B, int N, int k, uint8_t* flags,
                                  int* status, cudaStream_t s);
cudaError_t launch_gather(const void* src, int B, int N, int k, int row_bytes, const int32_t* idx,
                          void* dst, const int32_t* pos_in, int32_t* pos_out, int* status,
                          cudaStream_t s);
cudaError_t launch_rope_f32(float* qkv, int rows, int ld, int rope_cols, int hd,
                            const int32_t* pos, const float* cos_t, const float* sin_t,
                            cudaStream_t s);
cudaError_t launch_cls_head(int dtype, const void* h, int B, int N, int d, const void* norm_w,
                            float eps, const void* W, int n_classes, float* out, cudaStream_t s,
                            const int* cu = nullptr);  // cu: last row of b is cu[b+1]-1

// ---- GEMMs (k_gemm_tc.cu, k_gemm_simt.cu)
enum Epilogue : int { kEpiStore = 0, kEpiResid = 1, kEpiSwiGLU = 2, kEpiStoreF32 = 3, kEpiRope = 4 };

struct GemmParams {
  int M, N, K;
  void* out;            // [M, ldo] (N columns used; SwiGLU: N = output columns)
  int ldo;
  const void* resid;    // kEpiResid: [M, ldo]
  const int32_t* pos;   // kEpiRope: position of each row
  const float* cos_t;   // kEpiRope: [positions, hd/2]
  const float* sin_t;
  int rope_cols;        // kEpiRope: columns [0, rope_cols) are rotated
  int hd;               // kEpiRope: head size
  int* status;          // device status word
  float* splitk_ws;     // optional fp32 workspace for split tiles (NULL: whole tiles only)
  size_t splitk_ws_elems;
  int* splitk_flags;    // kMaxGemmCtas * 4 ints, zero before the first launch
  int* launches;        // optional host counter: kernels launched are added to it
  float* vnorm_out;     // kEpiRope: if set, ||v|| of each row's value heads, [M, (N - rope_cols) / hd]
};

// Stream-K workspace a caller should provide: one 128 x 256 fp32 tile per CTA
// (at most kMaxGemmCtas CTAs; the pair kernel counts both CTAs of a pair), and
// 4 flags per CTA.
constexpr int kMaxGemmCtas = 256;
constexpr size_t kSplitKWorkspaceElems = static_cast<size_t>(kMaxGemmCtas) * 128 * 256;
constexpr size_t kSplitKFlags = static_cast<size_t>(kMaxGemmCtas) * 4;

// bf16 tensor-core GEMM: out = epi(A[M,K] * W^T).  W is given as up to three
// row blocks (w0: rows [0, n1), w1: rows [n1, n2), w2: rows [n2, N)) so the
// QKV projection reads separate Wq/Wk/Wv; SwiGLU passes gate in w0 and up in
// w1 with n1 = N.
struct TcWeights {
  const void* w0;
  const void* w1;
  const void* w2;
  int n1, n2;
};
// Routing by rows: up to kSkinnyMaxM the weight-streaming kernel; up to the
// swap_preferred limit the swapped-operand kernel; else the persistent tiled
// kernel (k_gemm_tc.cu) on one CTA per SM, or on clusters of two CTAs sharing
// 256 x 256 tiles through the 2-SM MMA where that saves waves or splits a deep
// K (ZSAA_GEMM_PAIRS=0 in the environment keeps one CTA).
cudaError_t launch_gemm_tc(const void* A, int lda, const TcWeights& W, int epi,
                           const GemmParams& p, cudaStream_t s);
// The tiled kernels' plan for one call shape, computed on the host exactly as
// launch_gemm_tc computes it, for a device running `sms` CTAs and
// `pair_slots` CTA pairs at once and `split_slots` split-K partial slots
// (one weight matrix; RoPE heads of hd dims).  plan[12] and, up to cap of
// them, every unit's work items (8 ints each) in the order the unit runs
// them; *n_items = their number.  Returns 0; -1 when no tile width fits;
// -2 when the units' items outnumber the tiles' k-blocks (an iterator that
// does not advance).
int gemm_tc_schedule(int epi, int M, int N, int K, int hd, int sms, int pair_slots, int split_slots,
                     int* plan, int* items, long long cap, long long* n_items);

// Weight-streaming bf16 GEMM for M <= kSkinnyMaxM rows (k_skinny.cu): every
// epilogue but RoPE; N % 16 == 0, K % 32 == 0, lda % 8 == 0, 16-byte aligned
// A and W.  launch_gemm_tc routes such calls here.
constexpr int kSkinnyMaxM = 16;
bool skinny_supported(const void* A, int lda, const TcWeights& W, int epi, const GemmParams& p);
cudaError_t launch_gemm_skinny(const void* A, int lda, const TcWeights& W, int epi,
                               const GemmParams& p, cudaStream_t s);

// bf16 GEMM with the operands swapped (k_gemm_swap.cu) for kSkinnyMaxM < M <=
// kSwapMaxM: the weight band is the 128-row tcgen05 operand, the activation
// rows (blocks of at most kSwapRowBlock) the MMA's N side, and K is split over
// a thread-block cluster whose partial sums meet in distributed shared memory.
// Every epilogue; K % 64 == 0, N % 16 == 0, lda % 8 == 0, ldo % 4 == 0,
// 16-byte aligned pointers, weight row blocks on 128-row boundaries, RoPE with
// hd dividing 128.  launch_gemm_tc routes such calls here.
constexpr int kSwapMaxM = 1024;
constexpr int kSwapRowBlock = 256;
bool swap_supported(const void* A, int lda, const TcWeights& W, int epi, const GemmParams& p);
// Whether launch_gemm_tc takes the swapped kernel for this epilogue, row count
// and output width (wide float32 heads go to the tiled kernel).
bool swap_preferred(int epi, int M, int N, int K);
cudaError_t launch_gemm_swap(const void* A, int lda, const TcWeights& W, int epi,
                             const GemmParams& p, cudaStream_t s);

// fp32 CUDA-core GEMM, same epilogues (kEpiRope is applied by launch_rope_f32).
cudaError_t launch_gemm_f32(const float* A, int lda, const float* W, const float* W2, int epi,
                            const GemmParams& p, cudaStream_t s);

// ---- attention (k_attn.cu)
// Two-tile tcgen05 attention (k_attn_pp.cu) for bf16 heads of 64 or 128 dims,
// fixed lengths, an even number of query heads per KV head: persistent CTAs
// walk (sequence, KV group, pair of query heads, 128 queries) items, O kept
// in TMEM, V read from the qkv rows.  Same outputs as launch_attention;
// bounded waits report through status.
bool attention_pp_supported(int dtype, int hd, int Hq, int Hkv, const int* cu, const uint8_t* key_alive,
                            int* status);
cudaError_t launch_attention_pp(const void* qkv, int B, int N, int Hq, int Hkv, int hd, void* out, float* lse,
                                int causal, int* status, cudaStream_t s);
// tcgen05 attention (k_attn_tc.cu) for bf16 heads of 64 or 128 dims, fixed
// lengths: a transpose kernel writes V^T into vt (attention_tc_vt_elems bf16
// elements), then persistent CTAs walk (128 queries, head, sequence) items.
// Same outputs as launch_attention; bounded waits report through status.
bool attention_tc_supported(int dtype, int hd, const int* cu, const uint8_t* key_alive, int* status,
                            void* vt);
size_t attention_tc_vt_elems(int B, int N, int Hkv, int hd);
constexpr int kAttentionTcMinN = 256;
bool attention_tc_preferred(int N);
cudaError_t launch_attention_tc(const void* qkv, void* vt, int B, int N, int Hq, int Hkv, int hd, void* out,
                                float* lse, int causal, int* status, cudaStream_t s);
// causal = 0: bidirectional (Eq. 1 with M = 0); the column-mass kernels below
// take the same flag.
// cu (bf16 only): packed sequences of different lengths, rows [cu[b], cu[b+1]);
// N is then the longest length (grid size and the stride of lse).
cudaError_t launch_attention(int dtype, const void* qkv, int B, int N, int Hq, int Hkv, int hd,
                             void* out, float* lse, int causal, cudaStream_t s,
                             const int* cu = nullptr, const uint8_t* key_alive = nullptr);
// key_alive (bf16, fixed length): [B, N] flags of the masked mode; keys with 0
// are hidden from every query.
// Column mass C[B, Hkv, N] (via partial sums in `parts`, which must hold
// colmass_parts_elems(B, N, Hq, Hkv) floats).  bf16 with a status word runs
// the tensor-core kernel (k_colmass_tc.cu); otherwise the mma.sync / fp32 ones.
constexpr int kColmassQPer = 2;  // query blocks of 64 per mma.sync column-mass CTA
int colmass_chunks(int N);
size_t colmass_parts_elems(int B, int N, int Hq, int Hkv);
cudaError_t launch_colmass(int dtype, const void* qkv, const float* lse, int B, int N, int Hq,
                           int Hkv, int hd, float* parts, float* C, int* status, int causal,
                           cudaStream_t s);
// The score paths below take vnorm = ||v|| per row and group ([B*N, Hkv], from
// the QKV epilogue) for the bf16 tensor-core kernel; NULL makes the kernels
// compute the norms from qkv themselves.
// Position scores s[B, N] of R1 (mode ZSAA_SCORE_*): column mass weighted by
// ||v|| per group, summed over groups; same workspace as launch_colmass.
cudaError_t launch_position_scores(int dtype, const void* qkv, const float* lse, const float* vnorm,
                                   int B, int N, int Hq, int Hkv, int hd, int mode, float* parts,
                                   float* scores, int* status, int causal, cudaStream_t s);
// Only the partials of the position scores (for launch_select_parts); *n_qc
// receives the number of partial chunks.
cudaError_t launch_position_parts(int dtype, const void* qkv, const float* lse, const float* vnorm,
                                  int B, int N, int Hq, int Hkv, int hd, int mode, float* parts,
                                  int* n_qc, int* status, int causal, cudaStream_t s,
                                  const int* cu = nullptr, int rows = 0,
                                  const uint8_t* q_alive = nullptr);
// Tensor-core column-mass partials: parts[Hq/Hkv][B][Hkv][N] (per head of the
// group), times vnorm when it is not NULL; hd 64 or 128.  With cu: packed
// sequences of different lengths (rows [cu[b], cu[b+1]), `rows` in all, N the
// longest); vnorm is then per packed row.
cudaError_t launch_colmass_tc(const void* qkv, const float* lse, const float* vnorm, int B, int N,
                              int Hq, int Hkv, int hd, float* parts, int* status, int* n_chunks,
                              int causal, cudaStream_t s, const int* cu = nullptr, int rows = 0,
                              const uint8_t* q_alive = nullptr);

// ---- generation over the pruned KV cache (k_decode.cu)
// Cache of one layer: K and V bf16 [B, Hkv, cap, hd], positions int32 [B, cap].
struct KvLayer {
  void* k;  // bf16
  void* v;  // bf16
  int32_t* pos;
  int cap;   // rows per (sequence, group)
  int base;  // rows written by the prefill (N_{l-1})
};
// Prefill: copy the keys/values of the N rows per sequence in qkv (bf16,
// [B*N, ld], RoPE applied) and their positions into rows [0, N) of the cache.
cudaError_t launch_kv_write(const void* qkv, int ld, const int32_t* pos, int B, int N, int Hq,
                            int Hkv, int hd, const KvLayer& c, cudaStream_t s);
// One generated token per sequence: qkv32 [B, ld] float32 projections of the
// new rows; RoPE at position L0 + *step, bf16 rounding of q/k/v, k/v appended
// at cache row base + *step, then attention of the Hq queries over rows
// [0, base + *step]; out [B, Hq*hd] bf16.
cudaError_t launch_decode_attention(const float* qkv32, int ld, int B, int Hq, int Hkv, int hd,
                                    const KvLayer& c, const int* step, int L0, const float* cos_t,
                                    const float* sin_t, void* out, cudaStream_t s);
// *step += 1 (after every kernel of the decode step).
cudaError_t launch_decode_advance(int* step, cudaStream_t s);

// ---- thread-local message returned by zsaa_last_error (zsaa_api.cu)
void set_last_error(const char* msg);

// ---- driver entry point for tensor maps (zsaa_api.cu)
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn get_encode_tiled();

}  // namespace zsaa
