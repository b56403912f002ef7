/*
 * zsaa.h -- C ABI of the GB300 pruned-prefill library (Zero-Shot Adjustable
 * Acceleration, arXiv 2509.01190).
 *
 * The library runs the prefill forward pass of a pre-norm decoder (RMSNorm,
 * grouped-query attention with RoPE, SwiGLU MLP; Appendix A) in which, after
 * each pruning layer, every position is scored by its soft-score contribution
 * (Sec. 3.2-3.3), the top N_l positions are kept and compacted into a dense
 * [B, N_l, d] buffer, and the following layers run on those rows only.  N_l
 * follows Eq. 2 with a preservation rate alpha chosen per call from an
 * acceleration factor (Sec. 3.4).
 *
 * Conventions for every call:
 *  - Pointers documented "device" are CUDA device pointers; "host" pointers
 *    are ordinary CPU memory.  The library never frees caller memory.
 *  - Work is enqueued on the given stream and is asynchronous unless stated.
 *    Argument errors are found before anything is enqueued and return
 *    ZSAA_ERR_INVALID_ARG with nothing launched.
 *  - Device-side failures (a bounded wait that ran out) set a status word that
 *    zsaa_sync / zsaa_device_status report; kernels never trap.
 *  - No C++ exception crosses this boundary.  zsaa_last_error() returns a
 *    thread-local message for the last failing call on the calling thread.
 *  - Matrices are row-major.  Linear weights are [out_features, in_features]
 *    (each output feature's weights contiguous), the layout the GEMMs read as
 *    K-major operands.  bf16 buffers hold IEEE bfloat16 bit patterns.
 */
#ifndef ZSAA_H
#define ZSAA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#pragma GCC visibility push(default)
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* zsaa_stream;

typedef enum {
  ZSAA_OK = 0,
  ZSAA_ERR_INVALID_ARG = 1,
  ZSAA_ERR_OOM = 2,
  ZSAA_ERR_CUDA = 3,
  ZSAA_ERR_TIMEOUT = 4,
  ZSAA_ERR_UNSUPPORTED = 5
} zsaa_status;

/* Storage type of weights and activations. */
enum { ZSAA_F32 = 0, ZSAA_BF16 = 1 };

/* Position score (Sec. 3.2: soft-score times V is each V row's contribution).
 * SOFTSCORE_VNORM: s_j = sum_g C[g,j] * ||v_{g,j}||_2 ; SOFTSCORE: sum_g C[g,j]
 * where C[g,j] sums soft-score column j over all queries and over the query
 * heads of KV group g. */
enum { ZSAA_SCORE_SOFTSCORE_VNORM = 0, ZSAA_SCORE_SOFTSCORE = 1 };

/* Acceleration factor -> preservation rate (Sec. 3.4).  COST: the largest
 * alpha (60-step bisection on [0,1]) whose modelled per-sequence FLOPs are at
 * most 1/accel of the unpruned ones.  RATE: alpha = 1/accel. */
enum { ZSAA_PLAN_COST = 0, ZSAA_PLAN_RATE = 1 };

/* Flags of zsaa_score_select_ex. */
enum { ZSAA_FLAG_FORCE_KEEP_LAST = 1 };

/* Decoder shape and pruning options (Appendix A, Table 1; Eq. 2). */
typedef struct {
  int n_layers;     /* 1..64 */
  int d_model;      /* multiple of 64 */
  int n_heads;      /* query heads */
  int n_kv_heads;   /* KV heads; n_heads % n_kv_heads == 0 */
  int head_dim;     /* 32, 64 or 128 (bf16: 64 or 128) */
  int ffn_dim;      /* multiple of 64 */
  int vocab;        /* embedding rows */
  int n_classes;    /* 0: LM head over the vocabulary; >0: classifier on the last kept row */
  float rope_theta; /* RoPE base; frequency i of a head is theta^(-2i/head_dim) */
  float rms_eps;    /* RMSNorm epsilon */
  int dtype;        /* ZSAA_F32 or ZSAA_BF16 */
  int tau;          /* Eq. 2 floor on kept rows (the paper uses 5, Sec. 4.2) */
  uint64_t prune_mask;  /* bit l-1 set: layer l compacts its output rows */
  int force_keep_last;  /* 1: the last position is always kept (counts toward N_l) */
  int score_mode;       /* ZSAA_SCORE_* */
  int plan_mode;        /* ZSAA_PLAN_* */
  int bidirectional;    /* 0: causal decoder (Eq. 1 with the causal mask M); 1: encoder, M = 0 */
} zsaa_config;

/* Borrowed device weights; they must outlive the model.  layers points to a
 * HOST array of n_layers*9 device pointers, per layer in this order:
 *   attn_norm [d], wq [Hq*hd, d], wk [Hkv*hd, d], wv [Hkv*hd, d],
 *   wo [d, Hq*hd], mlp_norm [d], wg [F, d], wu [F, d], wd [d, F].
 * embed is [vocab, d]; final_norm [d]; head is [vocab, d] (may equal embed)
 * or [n_classes, d].  The pointer array itself is copied at create time. */
typedef struct {
  const void* embed;
  const void* const* layers;
  const void* final_norm;
  const void* head;
} zsaa_weights;

typedef struct zsaa_model zsaa_model;

/* Test and inspection hooks of zsaa_forward_ex.  All pointers are device
 * pointers or NULL.  Per-pruning-layer arrays are concatenated in layer order
 * over the layers whose bit is set in prune_mask (and that run):
 *   forced_idx : [B, N_l] int32 ascending indices into that layer's N_{l-1}
 *                rows, replacing the top-k choice (Sec. 3.3) there;
 *   scores_out : [B, N_{l-1}] float32 position scores of that layer;
 *   idx_out    : [B, N_l] int32 kept indices of that layer.
 * hidden_out : [B, N_last, d] residual rows leaving the last layer run.
 * n_layers_run: 0 runs through the last layer; m > 0 stops after layer m,
 *               then the head runs on the rows leaving layer m.
 * hidden_in  : [B, L, d] residual rows to start from instead of embedding
 *              token_ids (token_ids is then ignored and may be NULL); the
 *              pass starts at layer first_layer (1 .. n_layers + 1; n_layers
 *              + 1 runs only the head).  pos_in [B, L] gives the rows'
 *              original positions (NULL: 0..L-1).  The preservation rate is
 *              planned for sequences of plan_L tokens (0: L) and Eq. 2 is
 *              applied from N_{first_layer-1} = L. */
typedef struct {
  const int32_t* forced_idx;
  float* scores_out;
  int32_t* idx_out;
  void* hidden_out;
  int n_layers_run;
  const void* hidden_in;
  const int32_t* pos_in;
  int first_layer;
  int plan_L;
} zsaa_forward_opts;

/* Eq. 2 schedule for a config without a model (host only, no GPU needed).
 * n_sched receives N_0..N_{n_layers} (n_layers+1 ints, host); *alpha_out the
 * preservation rate.  accel >= 1; L >= 1. */
zsaa_status zsaa_plan_config(const zsaa_config* cfg, int L, double accel, int* n_sched,
                             double* alpha_out);

/* Validate the config, build GEMM tensor maps over the borrowed weights and
 * allocate workspace for batches up to max_B x max_L (device memory owned by
 * the model).  On error *out is NULL. */
zsaa_status zsaa_model_create(const zsaa_config* cfg, const zsaa_weights* w, int max_B,
                              int max_L, zsaa_model** out);

/* Free the model's workspace (not the weights).  Waits for the device. */
void zsaa_model_destroy(zsaa_model* m);

/* zsaa_plan_config for the model's config. */
zsaa_status zsaa_plan(const zsaa_model* m, int L, double accel, int* n_sched, double* alpha_out);

/* Pruned prefill of B sequences of L tokens (Sec. 3.3-3.4).
 *   token_ids   : device [B, L] int32 in [0, vocab)
 *   logits_out  : device float32 [B, N_final, vocab] (LM head; N_final is the
 *                 last entry of the schedule) or [B, n_classes]
 *   kept_pos_out: device int32 [B, N_final] original positions of the rows
 *                 the logits belong to, or NULL
 * 1 <= B <= max_B, 1 <= L <= max_L, accel >= 1. */
zsaa_status zsaa_forward(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                         float* logits_out, int32_t* kept_pos_out, zsaa_stream stream);

/* zsaa_forward and zsaa_forward_host replay repeated calls from CUDA graphs:
 * the first call with a given (token_ids, B, L, accel, logits_out,
 * kept_pos_out) runs eagerly, the second is captured on the given stream and
 * instantiated, and later ones launch the graph.  The 16 most recent argument
 * sets are kept per model.  A model is used by one host thread at a time.
 * zsaa_model_set_graphs(m, 0) turns this off (every call eager); 1 turns it
 * back on.  zsaa_forward_ex always runs eagerly. */
zsaa_status zsaa_model_set_graphs(zsaa_model* m, int enable);

/* zsaa_forward with the hooks of zsaa_forward_opts (opts may be NULL). */
zsaa_status zsaa_forward_ex(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                            float* logits_out, int32_t* kept_pos_out,
                            const zsaa_forward_opts* opts, zsaa_stream stream);

/* zsaa_forward on HOST buffers: copies token_ids (host [B, L]) in, runs, copies
 * logits (host float32, same shape as zsaa_forward) and kept positions (host or
 * NULL) out, and returns after the stream has finished.  Device staging is
 * owned by the model (allocated on first use).  When logits_out is page-locked
 * host memory (cudaHostAlloc / cudaHostRegister) and the model is a bf16 LM,
 * the LM head runs in column slabs and each slab is copied while the next one
 * computes; the values are the same either way. */
zsaa_status zsaa_forward_host(zsaa_model* m, const int32_t* token_ids, int B, int L,
                              double accel, float* logits_out, int32_t* kept_pos_out,
                              zsaa_stream stream);

/* zsaa_forward_masked: Appendix B's "marked, not removed" formulation as an
 * inference mode.  Every layer runs on all B*L rows; at a pruning layer the
 * scores come from the unmarked queries and keys, the top N_l unmarked rows
 * stay unmarked (Eq. 2 schedule, as zsaa_forward), and a marked row is hidden
 * as a key from every later layer.  Outputs have the layout of zsaa_forward
 * (logits of the final unmarked rows, their positions) and equal its values
 * up to rounding; the cost is that of the unpruned forward (nothing is
 * removed).  opts: NULL or the forced_idx / scores_out / idx_out hooks, with
 * indices given as POSITIONS [B, N_l] per pruning layer and scores [B, L] per
 * pruning layer (entries of marked rows unspecified); other fields zero.
 * bf16 models, d_model <= 4096, L <= 12288.  Row flags are owned by the
 * model (allocated on the first call). */
zsaa_status zsaa_forward_masked(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                                float* logits_out, int32_t* kept_pos_out,
                                const zsaa_forward_opts* opts, zsaa_stream stream);

/* zsaa_forward_marked: Appendix B's figure, where a row marked as pruned can
 * be reactivated at a later layer.  Reading: a row hidden as a key receives no
 * soft-score (Eq. 1) and so could never come back, so this mode hides and
 * removes nothing.  Every layer runs on all B*L rows exactly as the unpruned
 * forward does; each pruning layer marks as preserved the top N_l of ALL L
 * rows of each sequence by that layer's scores (Sec. 3.3 ranking, ties to the
 * lower position, the last position kept; N_l from the Eq. 2 schedule of
 * zsaa_plan), whatever the earlier marks.  Outputs: the logits of the rows
 * preserved at the last pruning layer (the unpruned forward's logits at those
 * positions) and their positions, laid out as zsaa_forward's.  opts as
 * zsaa_forward_masked (POSITIONS [B, N_l] and scores [B, L] per pruning layer).
 * Same limits as zsaa_forward_masked; the cost is that of the unpruned
 * forward plus the scoring of every pruning layer. */
zsaa_status zsaa_forward_marked(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                                float* logits_out, int32_t* kept_pos_out,
                                const zsaa_forward_opts* opts, zsaa_stream stream);

/* ---- Variable-length batches.
 *
 * Sec. 3.4 picks the preservation rate per inference call.  For one call over
 * sequences of different lengths the library reads it as one alpha for the
 * whole batch: ZSAA_PLAN_COST bisects (as zsaa_plan) for the largest alpha
 * whose modelled FLOPs summed over the batch are at most 1/accel of the
 * unpruned sum, and each sequence then follows Eq. 2 from its own length, so
 * sequence b keeps N_{l,b} rows after layer l.  ZSAA_PLAN_RATE: alpha = 1/accel.
 *
 * zsaa_plan_varlen(_config): lengths host int32 [B] (each >= 1); sched_out
 * host int [B][n_layers+1], row b = N_{0,b} .. N_{n,b}; alpha_out may be NULL.
 * Host only, no device work. */
zsaa_status zsaa_plan_varlen_config(const zsaa_config* cfg, const int32_t* lengths, int B,
                                    double accel, int* sched_out, double* alpha_out);
zsaa_status zsaa_plan_varlen(const zsaa_model* m, const int32_t* lengths, int B, double accel,
                             int* sched_out, double* alpha_out);

/* zsaa_forward_varlen: the pruned prefill of B sequences packed back to back.
 *   token_ids   : device int32 [T], T = sum of lengths, sequence b after b-1
 *   lengths     : host int32 [B], each in [1, max_L]; B <= max_B; T <= max_B*max_L
 *   logits_out  : device float32: LM head: the final kept rows of every
 *                 sequence, packed in order [sum_b N_{n,b}, vocab]; classifier:
 *                 [B, n_classes] from each sequence's last kept row
 *   kept_pos_out: device int32 [sum_b N_{n,b}] (positions within each sequence) or NULL
 *   opts        : NULL, or the forced_idx / scores_out / idx_out hooks of
 *                 zsaa_forward_ex with packed layouts: per pruning layer l,
 *                 indices [sum_b N_{l,b}] (within each sequence's rows) and
 *                 scores [sum_b N_{l-1,b}]; every other field zero.
 * A sequence attends only to its own rows.  bf16 models with d_model <= 4096
 * and lengths <= 12288 (ZSAA_ERR_UNSUPPORTED otherwise).  Runs eagerly; the
 * row offsets are uploaded from pinned memory the model owns (allocated on the
 * first call), and the call waits for the previous call's upload to finish. */
zsaa_status zsaa_forward_varlen(zsaa_model* m, const int32_t* token_ids, const int32_t* lengths,
                                int B, double accel, float* logits_out, int32_t* kept_pos_out,
                                const zsaa_forward_opts* opts, zsaa_stream stream);

/* ---- Generation over the pruned KV cache.
 *
 * Sec. 3.3 removes an eliminated row from every later layer, so after a pruned
 * prefill layer l holds the keys and values of only the N_{l-1} rows it ran
 * on.  A generated token attends, in layer l, to those rows, the tokens
 * generated before it and itself; generated tokens are never pruned.  The
 * cache therefore shrinks with depth like the prefill's rows do.
 *
 * zsaa_cache_create: a cache for B sequences of L prompt tokens pruned at
 * acceleration accel (the schedule of zsaa_plan), with room for max_new
 * generated tokens.  Layer l keeps cap_l = N_{l-1} + max_new rows per sequence
 * and KV group: K and V bf16 [B, Hkv, cap_l, hd] (keys after RoPE), positions
 * int32 [B, cap_l].  The cache belongs to the model's device and must not
 * outlive the model.  bf16 models with the language-model head and
 * force_keep_last set only (the last prompt position gives the first
 * generated token), else ZSAA_ERR_UNSUPPORTED.  B <= max_B, L <= max_L of the
 * model, max_new >= 1. */
typedef struct zsaa_cache zsaa_cache;
zsaa_status zsaa_cache_create(zsaa_model* m, int B, int L, double accel, int max_new,
                              zsaa_cache** out);
void zsaa_cache_destroy(zsaa_cache* c);

/* zsaa_prefill: the pruned prefill of zsaa_forward on token_ids (device int32
 * [B, L], the sizes the cache was made for) that also fills the cache, and
 * resets its generated count to 0.  logits_out: device float32 [B, V], the
 * logits of the last prompt position of each sequence (the next token).
 * opts may be NULL; its forced_idx / scores_out / idx_out hooks work as in
 * zsaa_forward_ex (the other fields must be zero). */
zsaa_status zsaa_prefill(zsaa_model* m, zsaa_cache* c, const int32_t* token_ids,
                         float* logits_out, const zsaa_forward_opts* opts, zsaa_stream stream);

/* zsaa_decode_step: one generated token per sequence.  token_ids: device int32
 * [B], the tokens at position L + t, where t = tokens generated since the
 * prefill (t < max_new, else ZSAA_ERR_INVALID_ARG; so is a call before the
 * first zsaa_prefill on the cache); logits_out: device float32
 * [B, V] for the next position.  Appends each layer's key and value to the
 * cache.  The position lives in device memory, so the step is recorded as a
 * CUDA graph on its second call with the same pointers and replayed after
 * that (zsaa_model_set_graphs controls this too). */
zsaa_status zsaa_decode_step(zsaa_model* m, zsaa_cache* c, const int32_t* token_ids,
                             float* logits_out, zsaa_stream stream);

/* zsaa_cache_layer: device pointers and sizes of layer l (1-based): k, v (bf16
 * [B, Hkv, cap, hd]), pos (int32 [B, cap]); *base = rows from the prefill
 * (N_{l-1}); *len = rows written so far (base + generated, counting steps
 * already enqueued).  Any out pointer may be NULL.  The pointers stay valid
 * for the cache's lifetime. */
zsaa_status zsaa_cache_layer(const zsaa_cache* c, int layer, void** k, void** v, int32_t** pos,
                             int* base, int* len, int* cap);

/* zsaa_cache_bytes: device bytes the cache holds for keys and values, and
 * what an unpruned cache (every layer L + max_new rows) would hold. */
zsaa_status zsaa_cache_bytes(const zsaa_cache* c, size_t* pruned, size_t* unpruned);

/* Isolated score + select + compaction (Sec. 3.3 with unit column mass and one
 * group, so the score of a row is its L2 norm):
 *   hidden      : device bf16 [B, L, d]
 *   idx_out     : device int32 [B, k], ascending kept indices per sequence
 *   gathered_out: device bf16 [B, k, d] kept rows, or NULL
 * 1 <= k <= L; d % 8 == 0.  Ties keep the lower index.  Scratch for the scores
 * is allocated stream-ordered from the device's default memory pool. */
zsaa_status zsaa_score_select(const void* hidden, int B, int L, int d, int k, int32_t* idx_out,
                              void* gathered_out, zsaa_stream stream);

/* zsaa_score_select with options: dtype ZSAA_BF16 or ZSAA_F32 rows; flags
 * ZSAA_FLAG_*; scores_in (device float32 [B, L]) replaces the computed scores
 * when not NULL; scores_out (device float32 [B, L]) receives the scores used.
 * NaN scores rank below every number. */
zsaa_status zsaa_score_select_ex(const void* hidden, int B, int L, int d, int dtype, int k,
                                 int flags, const float* scores_in, float* scores_out,
                                 int32_t* idx_out, void* gathered_out, zsaa_stream stream);

/* zsaa_score_select for callers that cannot allocate device memory while they
 * run (the paper has no counterpart; this is a property of the library).
 * Serving loops that reserve their memory budget up front, latency-critical
 * code that must avoid the allocator's locks and implicit synchronisation, and
 * hosts whose framework owns every device allocation cannot let a call take
 * scratch from the memory pool, as zsaa_score_select does for its B*L scores.
 * This call allocates nothing: the scores live in a fixed array of 1,048,576
 * floats (4 MiB) that the library holds on every GPU where its device code is
 * loaded, until the process exits.
 *   Arguments, layouts and results are those of zsaa_score_select.
 *   B*L above 1,048,576 is rejected with ZSAA_ERR_INVALID_ARG before any work.
 *   The first call on a device looks up the array's device address with that
 *   device current; make that first call before any stream capture.  The
 *   address is kept per device together with the id of the context it was
 *   found in; after a reset of that device's context (cudaDeviceReset) the
 *   next call looks it up again, so call once more outside capture then.
 *   All calls share the one array: calls whose work can overlap on the GPU
 *   (different streams, or different host threads) race on it and must be
 *   ordered by the caller. */
zsaa_status zsaa_score_select_noalloc(const void* hidden, int B, int L, int d, int k,
                                      int32_t* idx_out, void* gathered_out, zsaa_stream stream);

/* Single steps of the path, for per-kernel checks and timing.  All pointers
 * device; shapes as stated.
 * zsaa_op_linear: out[M,N] = epilogue(A[M,K] W[N,K]^T); dtype ZSAA_BF16 uses
 * the tcgen05 GEMMs (M <= 16 without RoPE: the weight-streaming GEMM; up to a
 * few hundred rows, by epilogue: the swapped-operand GEMM whose thread-block
 * cluster adds its split-K partials in a fixed order, so results do not depend
 * on timing; larger M: the persistent tiled GEMM, on clusters of two CTAs
 * sharing 256 x 256 tiles through the 2-SM MMA where that saves waves, its
 * split-K partials also added in a fixed order), ZSAA_F32 the fp32 CUDA-core
 * GEMM.  ZSAA_GEMM_PAIRS=0 in the environment (read once per process) keeps
 * the tiled GEMM on one CTA, a diagnostic switch with the same results up to
 * summation order.  The bf16 kernels start reading W before the
 * previous library kernel on the stream has finished: W and W2 must not be
 * written by that kernel.  epilogue:
 *   0 store (out has dtype; bf16 rounds once),
 *   1 residual: out = resid + acc (resid may alias out),
 *   2 SwiGLU: out[M,N] = silu(A W^T) * (A W2^T), W and W2 both [N,K],
 *   3 store float32 (out is float32 whatever dtype),
 *   4 RoPE: columns [0, rope_cols) are heads of rope_hd dims rotated at
 *     positions pos[M] (each in [0, 16384)) with base rope_theta
 *     (rotate-half pairing: dims c and c + rope_hd/2), then bf16 store.
 * K % 64 == 0 and N % 16 == 0 for bf16; RoPE only for bf16. */
zsaa_status zsaa_op_linear(const void* A, const void* W, const void* W2, const void* resid,
                           void* out, int M, int N, int K, int dtype, int epilogue,
                           const int32_t* pos, int rope_cols, int rope_hd, float rope_theta,
                           zsaa_stream stream);

/* The work decomposition of the persistent tiled GEMM (the kernel that
 * zsaa_op_linear and the forward use beyond the weight-streaming and
 * swapped-operand row ranges; the paper has no counterpart: this describes
 * how the library splits the projections of Appendix A over the device's SMs)
 * for one call shape, computed on the host exactly
 * as a launch computes it, without device work (no GPU needed).  The device
 * is described by sms (one-CTA kernel CTAs resident at once, one per SM;
 * >= 1), pair_slots (CTA pairs resident at once; 0: the pair kernel is not
 * used) and split_slots (split-K partial slots of 128 x 256 fp32 in the
 * workspace; 256 in the library's own workspaces, 0: no split).  One weight
 * matrix [N, K]; epilogue as zsaa_op_linear, RoPE heads of hd dims (hd >= 32,
 * a multiple of 32; other epilogues ignore hd).  K % 64 == 0, N % 16 == 0,
 * M >= 1.
 *   plan_out (host int32[12]): tile width, kernel (0 one CTA, 1 CTA pairs on
 *     256-row tiles), units (CTAs or pairs launched), row tiles, column tiles,
 *     64-deep k-blocks per tile, tiles, whole tiles dealt round robin first,
 *     k-iterations of the contiguous split that follows them, tiles of the
 *     aligned split (R) and their k-parts (S), 0.
 *   items (host int32[cap][8], or NULL with cap 0): every unit's work items
 *     in the order the unit runs them: unit, tile, first and end k-block, kind
 *     (0 a whole tile; 1 a part whose fp32 partial goes to slot `slot`; 2 the
 *     tile's final part, which waits for and adds the `count` partials in
 *     slots slot, slot + stride, ... in that order), slot, count, stride.
 *   *n_items (host) receives the number of items, including any past cap.
 * Unsupported shapes return ZSAA_ERR_INVALID_ARG or ZSAA_ERR_UNSUPPORTED; so
 * does a plan whose work items would outnumber its tiles' k-blocks (each item
 * covers at least one), which no sound plan has. */
zsaa_status zsaa_gemm_schedule(int epilogue, int M, int N, int K, int hd, int sms, int pair_slots,
                               int split_slots, int32_t* plan_out, int32_t* items, int64_t cap,
                               int64_t* n_items);

/* zsaa_op_attention: causal grouped-query attention (Eq. 1) over a packed
 * qkv [B*N, (Hq + 2 Hkv) hd] buffer (per row: Hq query heads, then Hkv key
 * heads, then Hkv value heads).  out [B*N, Hq*hd]; lse float32 [B, Hq, N]
 * gets log2 of the softmax normaliser of the scaled logits (log2 domain). */
zsaa_status zsaa_op_attention(const void* qkv, int B, int N, int Hq, int Hkv, int hd, int dtype,
                              void* out, float* lse, zsaa_stream stream);

/* zsaa_op_colmass: C[B, Hkv, N] float32, C[b,g,j] = sum over the query heads
 * of group g and queries i >= j of the soft-score P[i,j] (Sec. 3.2), using
 * the lse that zsaa_op_attention wrote. */
zsaa_status zsaa_op_colmass(const void* qkv, const float* lse, int B, int N, int Hq, int Hkv,
                            int hd, int dtype, float* colmass, zsaa_stream stream);

/* The two steps above with the mask of Eq. 1 chosen: causal = 1 as above,
 * causal = 0 for a bidirectional encoder (M = 0: every query sees every key,
 * and the column mass sums P[i,j] over all queries i). */
zsaa_status zsaa_op_attention_ex(const void* qkv, int B, int N, int Hq, int Hkv, int hd, int dtype,
                                 int causal, void* out, float* lse, zsaa_stream stream);
zsaa_status zsaa_op_colmass_ex(const void* qkv, const float* lse, int B, int N, int Hq, int Hkv,
                               int hd, int dtype, int causal, float* colmass, zsaa_stream stream);

/* Per-kernel timing of the forward pass.  After zsaa_trace_begin every
 * kernel the model launches is bracketed by CUDA events recorded on the launch
 * stream (this adds a small gap between launches, so traced forwards are not
 * for headline timing).  zsaa_trace_end waits for the device, stops recording
 * and fills up to max_rows rows (host array), one per kernel class in first
 * launch order: launches, summed device milliseconds, and the algorithmic
 * FLOPs (2 per multiply-add; causal attention counts only j <= i) and HBM
 * bytes (each tensor read or written once) of those launches. */
typedef struct {
  char name[32];
  int launches;
  double ms;
  double flops;
  double bytes;
} zsaa_trace_row;

zsaa_status zsaa_trace_begin(zsaa_model* m);
zsaa_status zsaa_trace_end(zsaa_model* m, zsaa_trace_row* rows, int max_rows, int* n_rows);

/* Wait for the stream and report the model's device status word (then clear
 * it): ZSAA_OK, or ZSAA_ERR_TIMEOUT if a kernel gave up a bounded wait. */
zsaa_status zsaa_sync(zsaa_model* m, zsaa_stream stream);

/* Status word shared by the calls that have no model (zsaa_score_select*,
 * zsaa_op_*): synchronises the device, returns it and clears it. */
zsaa_status zsaa_device_status(void);

/* Self-test of the device failure path (bounded waits that report a status,
 * never a trap: the error model above).  Launches on `stream` one CTA whose two roles wait,
 * with the same bounded mbarrier wait as every pipelined kernel, for a barrier
 * phase that nothing completes.  The wait gives up after its limit (2 s), sets
 * the timeout bit of the status word shared by the model-less calls, and the
 * kernel returns; the context stays usable.  Waits for the stream and returns
 * that status (then clears it): ZSAA_ERR_TIMEOUT when the path works, ZSAA_OK
 * if the wait ended some other way.  Takes about 2 s of GPU time. */
zsaa_status zsaa_selftest_wait_timeout(zsaa_stream stream);

/* Message of the last failing call on this thread ("" if none). */
const char* zsaa_last_error(void);

/* Library version string. */
const char* zsaa_version(void);

#if defined(__GNUC__)
#pragma GCC visibility pop
#endif

#ifdef __cplusplus
}
#endif

#endif /* ZSAA_H */
