// C ABI of the pruned-prefill library: planner (Eq. 2, Sec. 3.4), model
// workspace, and the stream-ordered forward pass that chains the kernels.
//
// Forward pass of one call (Sec. 3.3): embed -> for each layer l on N_{l-1}
// rows: RMSNorm, QKV GEMM with RoPE at original positions, causal GQA
// attention, O GEMM + residual; if layer l prunes and N_l < N_{l-1}: column
// mass, scores, top-k, gather of the residual rows and their positions; then
// RMSNorm, gate/up GEMM with SwiGLU, down GEMM + residual on the N_l kept rows
// (the MLP is row-wise, so compacting before it changes no kept row) -> final
// RMSNorm + head.
// The schedule is computed on the host before any launch; there is no
// host/device synchronisation inside a forward.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <list>
#include <mutex>
#include <string>
#include <unordered_map>
#include <vector>

#include "common.cuh"
#include "kernels.h"

using namespace zsaa;

namespace {

thread_local std::string g_last_error;

zsaa_status fail(zsaa_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

#define ZCK(expr)                                                                        \
  do {                                                                                   \
    cudaError_t e_ = (expr);                                                             \
    if (e_ != cudaSuccess)                                                               \
      return fail(ZSAA_ERR_CUDA, "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), \
                  __FILE__, __LINE__);                                                   \
  } while (0)

// ---------------------------------------------------------------- planner

bool prunes(const zsaa_config& c, int layer) { return (c.prune_mask >> (layer - 1)) & 1ull; }

// Eq. 2: N_l = min(N_{l-1}, max(floor(alpha N_{l-1}), min(tau, N_{l-1}))) after a pruning layer.
void eq2_schedule(const zsaa_config& c, int L, double alpha, int* out) {
  out[0] = L;
  for (int l = 1; l <= c.n_layers; ++l) {
    const int prev = out[l - 1];
    if (prunes(c, l)) {
      long long nl = static_cast<long long>(std::floor(alpha * static_cast<double>(prev)));
      const long long floor_rows = prev < c.tau ? prev : c.tau;
      if (nl < floor_rows) nl = floor_rows;
      out[l] = static_cast<int>(nl < prev ? nl : prev);
    } else {
      out[l] = prev;
    }
  }
}

// Modelled FLOPs of one sequence: linear layers + causal attention + head.
long long model_cost(const zsaa_config& c, const int* sched) {
  const long long d = c.d_model, hd = c.head_dim, dq = static_cast<long long>(c.n_heads) * hd;
  const long long f = 2 * d * (dq + 2LL * c.n_kv_heads * hd) + 2 * dq * d + 6 * d * c.ffn_dim;
  long long total = 0;
  for (int l = 0; l < c.n_layers; ++l) {
    const long long n = sched[l];
    total += n * f + 2 * n * n * dq;
  }
  if (c.n_classes > 0)
    total += 2 * d * c.n_classes;
  else
    total += static_cast<long long>(sched[c.n_layers]) * 2 * d * c.vocab;
  return total;
}

zsaa_status plan_impl(const zsaa_config& c, int L, double accel, int* sched, double* alpha_out) {
  if (!(accel >= 1.0)) return fail(ZSAA_ERR_INVALID_ARG, "accel must be >= 1 (got %g)", accel);
  if (L < 1) return fail(ZSAA_ERR_INVALID_ARG, "L must be >= 1");
  double alpha = 1.0;
  if (c.plan_mode == ZSAA_PLAN_RATE) {
    alpha = 1.0 / accel;
  } else if (accel != 1.0) {
    std::vector<int> s(c.n_layers + 1);
    eq2_schedule(c, L, 1.0, s.data());
    const double target = static_cast<double>(model_cost(c, s.data())) / accel;
    double lo = 0.0, hi = 1.0;
    for (int it = 0; it < 60; ++it) {
      const double mid = 0.5 * (lo + hi);
      eq2_schedule(c, L, mid, s.data());
      if (static_cast<double>(model_cost(c, s.data())) <= target)
        lo = mid;
      else
        hi = mid;
    }
    alpha = lo;
  }
  eq2_schedule(c, L, alpha, sched);
  if (alpha_out) *alpha_out = alpha;
  return ZSAA_OK;
}

// One rate for B sequences of different lengths (R17): the "cost" mode bisects
// on the modelled FLOPs summed over the batch; each sequence then follows
// Eq. 2 from its own length.  sched: [B][n_layers + 1].  Sums stay exact
// integers below 2^53, so the oracle's planner agrees bit for bit.
zsaa_status plan_varlen_impl(const zsaa_config& c, const int32_t* lengths, int B, double accel,
                             int* sched, double* alpha_out) {
  if (!(accel >= 1.0)) return fail(ZSAA_ERR_INVALID_ARG, "accel must be >= 1 (got %g)", accel);
  if (B < 1 || lengths == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "need B >= 1 lengths");
  for (int b = 0; b < B; ++b)
    if (lengths[b] < 1) return fail(ZSAA_ERR_INVALID_ARG, "length %d of sequence %d is < 1", lengths[b], b);
  const int n1 = c.n_layers + 1;
  auto fill = [&](double a) {
    long long total = 0;
    for (int b = 0; b < B; ++b) {
      eq2_schedule(c, lengths[b], a, sched + static_cast<size_t>(b) * n1);
      total += model_cost(c, sched + static_cast<size_t>(b) * n1);
    }
    return total;
  };
  double alpha = 1.0;
  if (c.plan_mode == ZSAA_PLAN_RATE) {
    alpha = 1.0 / accel;
  } else if (accel != 1.0) {
    const double target = static_cast<double>(fill(1.0)) / accel;
    double lo = 0.0, hi = 1.0;
    for (int it = 0; it < 60; ++it) {
      const double mid = 0.5 * (lo + hi);
      if (static_cast<double>(fill(mid)) <= target)
        lo = mid;
      else
        hi = mid;
    }
    alpha = lo;
  }
  fill(alpha);
  if (alpha_out) *alpha_out = alpha;
  return ZSAA_OK;
}

zsaa_status validate_config(const zsaa_config& c) {
  if (c.n_layers < 1 || c.n_layers > 64) return fail(ZSAA_ERR_INVALID_ARG, "n_layers must be 1..64");
  if (c.dtype != ZSAA_F32 && c.dtype != ZSAA_BF16) return fail(ZSAA_ERR_INVALID_ARG, "bad dtype");
  if (c.n_heads < 1 || c.n_kv_heads < 1 || c.n_heads % c.n_kv_heads != 0)
    return fail(ZSAA_ERR_INVALID_ARG, "n_heads must be a positive multiple of n_kv_heads");
  if (c.head_dim < 2 || c.head_dim % 2 != 0 || c.head_dim > 128)
    return fail(ZSAA_ERR_INVALID_ARG, "head_dim must be even and <= 128");
  if (c.d_model < 8 || c.d_model % 8 != 0 || c.ffn_dim < 1 || c.vocab < 1)
    return fail(ZSAA_ERR_INVALID_ARG, "bad d_model / ffn_dim / vocab");
  if (c.tau < 1) return fail(ZSAA_ERR_INVALID_ARG, "tau must be >= 1");
  if (c.n_classes < 0) return fail(ZSAA_ERR_INVALID_ARG, "n_classes must be >= 0");
  if (c.score_mode != ZSAA_SCORE_SOFTSCORE_VNORM && c.score_mode != ZSAA_SCORE_SOFTSCORE)
    return fail(ZSAA_ERR_INVALID_ARG, "bad score_mode");
  if (c.plan_mode != ZSAA_PLAN_COST && c.plan_mode != ZSAA_PLAN_RATE)
    return fail(ZSAA_ERR_INVALID_ARG, "bad plan_mode");
  if (c.bidirectional != 0 && c.bidirectional != 1) return fail(ZSAA_ERR_INVALID_ARG, "bidirectional must be 0 or 1");
  if (c.n_layers < 64 && (c.prune_mask >> c.n_layers) != 0)
    return fail(ZSAA_ERR_INVALID_ARG, "prune_mask names layers beyond n_layers");
  if (c.dtype == ZSAA_BF16) {
    const int dq = c.n_heads * c.head_dim;
    if (c.head_dim != 64 && c.head_dim != 128)
      return fail(ZSAA_ERR_UNSUPPORTED, "bf16 models need head_dim 64 or 128");
    if (c.d_model % 64 || dq % 64 || c.ffn_dim % 64)
      return fail(ZSAA_ERR_UNSUPPORTED, "bf16 models need d_model, heads*head_dim, ffn_dim % 64 == 0");
    if ((c.n_kv_heads * c.head_dim) % 64)
      return fail(ZSAA_ERR_UNSUPPORTED, "bf16 models need kv_heads*head_dim % 64 == 0");
    if (c.n_classes == 0 && c.vocab % 16)
      return fail(ZSAA_ERR_UNSUPPORTED, "bf16 LM head needs vocab % 16 == 0");
  } else if (c.d_model % 4) {
    return fail(ZSAA_ERR_UNSUPPORTED, "f32 models need d_model % 4 == 0");
  }
  return ZSAA_OK;
}

// ---------------------------------------------------------------- device helpers

EncodeTiledFn g_encode = nullptr;
std::once_flag g_encode_once;

std::mutex g_status_mu;
std::unordered_map<int, int*> g_status_by_dev;  // shared status word of model-less calls

int* shared_status() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  std::lock_guard<std::mutex> lk(g_status_mu);
  auto it = g_status_by_dev.find(dev);
  if (it != g_status_by_dev.end()) return it->second;
  int* p = nullptr;
  if (cudaMalloc(&p, sizeof(int)) != cudaSuccess) return nullptr;
  if (cudaMemset(p, 0, sizeof(int)) != cudaSuccess) {
    cudaFree(p);
    return nullptr;
  }
  g_status_by_dev[dev] = p;
  return p;
}

// Split-K workspace of zsaa_op_linear, one per device, allocated on first use.
std::mutex g_ws_mu;
std::unordered_map<int, std::pair<float*, int*>> g_op_ws;

bool op_splitk_ws(float** ws, int** flags) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  std::lock_guard<std::mutex> lk(g_ws_mu);
  auto it = g_op_ws.find(dev);
  if (it == g_op_ws.end()) {
    float* p = nullptr;
    int* f = nullptr;
    if (cudaMalloc(&p, kSplitKWorkspaceElems * sizeof(float)) != cudaSuccess) return false;
    if (cudaMalloc(&f, kSplitKFlags * sizeof(int)) != cudaSuccess ||
        cudaMemset(f, 0, kSplitKFlags * sizeof(int)) != cudaSuccess) {
      cudaFree(p);
      if (f != nullptr) cudaFree(f);
      return false;
    }
    it = g_op_ws.emplace(dev, std::make_pair(p, f)).first;
  }
  *ws = it->second.first;
  *flags = it->second.second;
  return true;
}

// RoPE tables of zsaa_op_linear, cached per (device, theta, head size):
// positions 0 .. kOpRopePositions-1.
constexpr int kOpRopePositions = 16384;
struct RopeTable {
  float* cos_t;
  float* sin_t;
};
std::mutex g_rope_mu;
std::unordered_map<std::string, RopeTable> g_rope_tables;

bool op_rope_table(float theta, int hd, RopeTable* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  char key[96];
  snprintf(key, sizeof(key), "%d/%.9g/%d", dev, static_cast<double>(theta), hd);
  std::lock_guard<std::mutex> lk(g_rope_mu);
  auto it = g_rope_tables.find(key);
  if (it != g_rope_tables.end()) {
    *out = it->second;
    return true;
  }
  const int half = hd / 2;
  std::vector<float> c(static_cast<size_t>(kOpRopePositions) * half), sv(c.size());
  for (int q = 0; q < kOpRopePositions; ++q)
    for (int i = 0; i < half; ++i) {
      const double a = static_cast<double>(q) *
                       std::pow(static_cast<double>(theta), -2.0 * i / static_cast<double>(hd));
      c[static_cast<size_t>(q) * half + i] = static_cast<float>(std::cos(a));
      sv[static_cast<size_t>(q) * half + i] = static_cast<float>(std::sin(a));
    }
  RopeTable t{nullptr, nullptr};
  const bool ok = cudaMalloc(&t.cos_t, c.size() * 4) == cudaSuccess &&
                  cudaMalloc(&t.sin_t, c.size() * 4) == cudaSuccess &&
                  cudaMemcpy(t.cos_t, c.data(), c.size() * 4, cudaMemcpyHostToDevice) == cudaSuccess &&
                  cudaMemcpy(t.sin_t, sv.data(), c.size() * 4, cudaMemcpyHostToDevice) == cudaSuccess;
  if (!ok) {
    if (t.cos_t != nullptr) cudaFree(t.cos_t);
    if (t.sin_t != nullptr) cudaFree(t.sin_t);
    return false;
  }
  g_rope_tables[key] = t;
  *out = t;
  return true;
}

}  // namespace

namespace zsaa {
void set_last_error(const char* msg) { g_last_error = msg; }

EncodeTiledFn get_encode_tiled() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<EncodeTiledFn>(fn);
  });
  return g_encode;
}
}  // namespace zsaa

// ---------------------------------------------------------------- model

struct zsaa_model {
  zsaa_config cfg;
  int max_B = 0, max_L = 0;
  int device = 0;
  const void* embed = nullptr;
  const void* final_norm = nullptr;
  const void* head = nullptr;
  std::vector<const void*> layers;  // n_layers * 9
  size_t esz = 2;
  int ld_qkv = 0, dq = 0, dkv = 0;
  // workspace
  void* h[2] = {nullptr, nullptr};
  void* x = nullptr;
  void* qkv = nullptr;
  void* attn = nullptr;
  void* act = nullptr;
  float* lse = nullptr;
  void* vt = nullptr;        // V^T of the current layer for the tcgen05 attention (bf16, hd 64)
  float* colmass = nullptr;  // query-chunk partials of the column mass / scores
  float* vnorm = nullptr;    // ||v|| per row and KV group, from the QKV epilogue (bf16)
  float* scores = nullptr;
  int32_t* idx = nullptr;
  int32_t* pos[2] = {nullptr, nullptr};
  float* rope_cos = nullptr;
  float* rope_sin = nullptr;
  float* splitk_ws = nullptr;
  int* splitk_flags = nullptr;
  int* status = nullptr;
  // host-buffer staging (zsaa_forward_host)
  int32_t* stage_tok = nullptr;
  float* stage_logits = nullptr;
  int32_t* stage_pos = nullptr;
  size_t stage_logits_cap = 0;
  // packed-sequence row offsets of zsaa_forward_varlen (device, and the pinned
  // host copy they are uploaded from; the event guards its reuse)
  uint8_t* alive = nullptr;  // masked mode: [max_B, max_L] row flags (allocated on first use)
  int32_t* vl_cu = nullptr;
  int32_t* vl_cu_host = nullptr;
  cudaEvent_t vl_done = nullptr;
  // tracing (zsaa_trace_begin / _end)
  struct TraceRec {
    int cls;
    int kernels;
    cudaEvent_t a, b;
    double flops, bytes;
  };
  bool tracing = false;
  std::vector<TraceRec> trace;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  std::vector<std::string> trace_names;
  // CUDA graphs of plain forwards, keyed by their arguments (most recent first)
  struct GraphEntry {
    std::string key;
    int seen = 0;                 // eager runs so far with this key
    cudaGraphExec_t exec = nullptr;
    const void* cache = nullptr;  // zsaa_cache whose buffers the graph uses, if any
  };
  bool use_graphs = true;
  std::list<GraphEntry> graphs;
  cudaStream_t capture_stream = nullptr;  // graphs are recorded here, launched on the caller's
  // side stream of a pruning layer's O-projection (forked after the attention,
  // joined before the gather), created on first use
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // zsaa_forward_host with a pinned logits buffer: the LM head runs in column
  // slabs and each slab is copied to this host buffer while the next computes
  float* host_logits = nullptr;
};

// Pruned KV cache for generation (zsaa_cache_create).
struct zsaa_cache {
  zsaa_model* m = nullptr;
  int B = 0, L = 0, max_new = 0;
  double accel = 1.0, alpha = 1.0;
  std::vector<int> sched;                // N_0 .. N_n
  std::vector<zsaa::KvLayer> layers;     // per layer (0-based)
  void* kv = nullptr;                    // every layer's K then V
  int32_t* pos = nullptr;                // every layer's positions
  size_t kv_bytes = 0, kv_bytes_unpruned = 0;
  float* rope_cos = nullptr;             // [L + max_new, hd/2]
  float* rope_sin = nullptr;
  float* qkv32 = nullptr;                // [B, ld_qkv] float32 projections of the new rows
  int32_t* last_idx = nullptr;           // [B]: N_n - 1, the last kept row
  int* step = nullptr;                   // device: tokens generated since the prefill
  int generated = 0;                     // host: decode steps enqueued since the prefill
  bool prefilled = false;                // a prefill has been enqueued
  // CUDA graph of the decode step, keyed by its pointers
  std::string graph_key;
  int graph_seen = 0;
  cudaGraphExec_t graph = nullptr;
};

namespace {

// Column slabs of the LM head when its logits stream to a pinned host buffer
// (zsaa_forward_host): slab i covers columns [slab_col(V, i), slab_col(V, i+1)),
// boundaries on 128-column multiples.
constexpr int kHeadSlabs = 4;
int slab_col(int V, int i, int n) {
  if (i >= n) return V;
  const long long c = (static_cast<long long>(V) * i / n + 127) / 128 * 128;
  return static_cast<int>(c < V ? c : V);
}

// Make the model's side stream wait for the work enqueued on s so far
// (creating the stream and its events on first use).
cudaError_t fork_side(zsaa_model* m, cudaStream_t s) {
  if (m->side == nullptr) {
    cudaError_t e = cudaStreamCreateWithFlags(&m->side, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&m->ev_fork, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&m->ev_join, cudaEventDisableTiming);
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = cudaEventRecord(m->ev_fork, s);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(m->side, m->ev_fork, 0);
  return e;
}

const void* LW(const zsaa_model* m, int layer, int slot) {
  return m->layers[static_cast<size_t>(layer) * 9 + slot];
}
enum { kAttnNorm = 0, kWq, kWk, kWv, kWo, kMlpNorm, kWg, kWu, kWd };

// Brackets one kernel launch with events while the model is tracing.
class TraceScope {
 public:
  TraceScope(zsaa_model* m, const char* name, double flops, double bytes, cudaStream_t s)
      : m_(m), s_(s) {
    if (!m->tracing) return;
    int cls = -1;
    for (size_t i = 0; i < m->trace_names.size(); ++i)
      if (m->trace_names[i] == name) cls = static_cast<int>(i);
    if (cls < 0) {
      cls = static_cast<int>(m->trace_names.size());
      m->trace_names.push_back(name);
    }
    rec_.cls = cls;
    rec_.flops = flops;
    rec_.bytes = bytes;
    rec_.a = event();
    rec_.b = event();
    if (rec_.a && rec_.b && cudaEventRecord(rec_.a, s) == cudaSuccess) active_ = true;
  }
  ~TraceScope() {
    rec_.kernels = kernels;
    if (active_ && cudaEventRecord(rec_.b, s_) == cudaSuccess) m_->trace.push_back(rec_);
  }
  int kernels = 1;  // kernels launched inside the scope

 private:
  cudaEvent_t event() {
    if (m_->ev_used == m_->ev_pool.size()) {
      cudaEvent_t e = nullptr;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      m_->ev_pool.push_back(e);
    }
    return m_->ev_pool[m_->ev_used++];
  }
  zsaa_model* m_;
  cudaStream_t s_;
  zsaa_model::TraceRec rec_{};
  bool active_ = false;
};

void free_model(zsaa_model* m) {
  if (m == nullptr) return;
  for (cudaEvent_t e : m->ev_pool) cudaEventDestroy(e);
  for (auto& g : m->graphs)
    if (g.exec) cudaGraphExecDestroy(g.exec);
  if (m->capture_stream) cudaStreamDestroy(m->capture_stream);
  if (m->side) cudaStreamDestroy(m->side);
  if (m->ev_fork) cudaEventDestroy(m->ev_fork);
  if (m->ev_join) cudaEventDestroy(m->ev_join);
  void* ptrs[] = {m->h[0], m->h[1], m->x, m->qkv, m->attn, m->act, m->lse, m->vt, m->colmass, m->vnorm,
                  m->scores, m->idx, m->pos[0], m->pos[1], m->rope_cos, m->rope_sin,
                  m->splitk_ws, m->splitk_flags, m->status, m->stage_tok, m->stage_logits,
                  m->stage_pos};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  if (m->vl_cu) cudaFree(m->vl_cu);
  if (m->alive) cudaFree(m->alive);
  if (m->vl_cu_host) cudaFreeHost(m->vl_cu_host);
  if (m->vl_done) cudaEventDestroy(m->vl_done);
  delete m;
}

// out[M, N] = epi(A W^T) on the model's dtype path.
zsaa_status linear(zsaa_model* m, const void* A, int lda, const TcWeights& W, int epi,
                   GemmParams p, cudaStream_t s, int* kernels = nullptr) {
  p.status = m->status;
  p.splitk_ws = m->splitk_ws;
  p.splitk_ws_elems = m->splitk_ws ? kSplitKWorkspaceElems : 0;
  p.splitk_flags = m->splitk_flags;
  p.launches = kernels;
  if (m->cfg.dtype == ZSAA_BF16) {
    ZCK(launch_gemm_tc(A, lda, W, epi, p, s));
  } else {
    if (epi == kEpiRope) return fail(ZSAA_ERR_UNSUPPORTED, "f32 RoPE epilogue");
    ZCK(launch_gemm_f32(static_cast<const float*>(A), lda, static_cast<const float*>(W.w0),
                        static_cast<const float*>(W.w1), epi, p, s));
  }
  return ZSAA_OK;
}

// With a cache (zsaa_prefill) every layer's keys/values are copied into it and
// only the last kept row of each sequence goes through the head.
zsaa_status run_forward(zsaa_model* m, const int32_t* tok, int B, int L, double accel,
                        float* logits, int32_t* kept_pos, const zsaa_forward_opts* opts,
                        cudaStream_t s, zsaa_cache* kc = nullptr) {
  const zsaa_config& c = m->cfg;
  const bool from_hidden = opts && opts->hidden_in;
  if ((!from_hidden && tok == nullptr) || logits == nullptr)
    return fail(ZSAA_ERR_INVALID_ARG, "null token or logits pointer");
  if (B < 1 || B > m->max_B || L < 1 || L > m->max_L)
    return fail(ZSAA_ERR_INVALID_ARG, "B=%d L=%d outside [1,%d] x [1,%d]", B, L, m->max_B, m->max_L);
  const int first = from_hidden ? opts->first_layer : 1;
  const int n_run = (opts && opts->n_layers_run > 0) ? opts->n_layers_run : c.n_layers;
  if (first < 1 || first > c.n_layers + 1) return fail(ZSAA_ERR_INVALID_ARG, "first_layer outside [1, n_layers+1]");
  if (n_run > c.n_layers || n_run < first - 1) return fail(ZSAA_ERR_INVALID_ARG, "bad n_layers_run");
  const int plan_L = (from_hidden && opts->plan_L > 0) ? opts->plan_L : L;
  std::vector<int> sched(c.n_layers + 1);
  double alpha = 1.0;
  zsaa_status st = plan_impl(c, plan_L, accel, sched.data(), &alpha);
  if (st != ZSAA_OK) return st;
  if (from_hidden) {  // Eq. 2 continued from the rows given
    sched[first - 1] = L;
    for (int l = first; l <= c.n_layers; ++l) {
      int tmp[2];
      zsaa_config one = c;
      one.n_layers = 1;
      one.prune_mask = prunes(c, l) ? 1ull : 0ull;
      eq2_schedule(one, sched[l - 1], alpha, tmp);
      sched[l] = tmp[1];
    }
  }

  const int d = c.d_model, hd = c.head_dim, Hq = c.n_heads, Hkv = c.n_kv_heads;
  const int dt = c.dtype;
  const int causal = c.bidirectional ? 0 : 1;
  // query-key pairs of Eq. 1 per sequence and head
  auto n_pairs = [&](int n) { return causal ? static_cast<double>(n) * (n + 1) / 2.0 : static_cast<double>(n) * n; };
  int cur = 0;
  const double es = static_cast<double>(m->esz);
#define TRACE(name, fl, by) TraceScope trace_scope_(m, name, fl, by, s)
  if (from_hidden) {
    ZCK(cudaMemcpyAsync(m->h[cur], opts->hidden_in, static_cast<size_t>(B) * L * d * m->esz,
                        cudaMemcpyDeviceToDevice, s));
    if (opts->pos_in) {
      ZCK(cudaMemcpyAsync(m->pos[cur], opts->pos_in, sizeof(int32_t) * B * L,
                          cudaMemcpyDeviceToDevice, s));
    } else {
      std::vector<int32_t> iota(static_cast<size_t>(B) * L);
      for (size_t i = 0; i < iota.size(); ++i) iota[i] = static_cast<int32_t>(i % L);
      ZCK(cudaMemcpyAsync(m->pos[cur], iota.data(), iota.size() * sizeof(int32_t),
                          cudaMemcpyHostToDevice, s));
      ZCK(cudaStreamSynchronize(s));
    }
  }
  // bf16 rows of moderate width: embedding and compaction also write the next
  // layer's normed input (x_ready), saving that layer's RMSNorm launch.
  const bool fuse_norm = dt == ZSAA_BF16 && d % 8 == 0 && d <= kRowsNormMaxD;
  bool x_ready = false;
  if (!from_hidden) {
    if (fuse_norm && first <= n_run) {
      TRACE("embed_norm", 0.0, static_cast<double>(B) * L * (3.0 * d * es + 8.0));
      ZCK(launch_rows_norm(m->embed, tok, c.vocab, L, nullptr, 0, 0, nullptr, B * L, d,
                           LW(m, first - 1, kAttnNorm), c.rms_eps, m->h[cur], m->x, m->pos[cur],
                           m->status, s));
      x_ready = true;
    } else {
      TRACE("embed", 0.0, static_cast<double>(B) * L * (d * es + 8.0));
      ZCK(launch_embed(dt, m->embed, tok, B * L, L, c.vocab, d, m->h[cur], m->pos[cur], m->status, s));
    }
  }
  size_t off_forced = 0, off_scores = 0, off_idx = 0;
  int N = L;
  for (int l = first; l <= n_run; ++l) {
    const int li = l - 1;
    const int M = B * N;
    void* h = m->h[cur];
    const double Md = static_cast<double>(M);
    // attention branch
    if (!x_ready) {
      TRACE("rmsnorm", 0.0, 2.0 * Md * d * es);
      ZCK(launch_rmsnorm(dt, h, LW(m, li, kAttnNorm), M, d, c.rms_eps, m->x, s));
    }
    x_ready = false;
    GemmParams p{};
    p.M = M;
    p.K = d;
    p.out = m->qkv;
    p.ldo = m->ld_qkv;
    if (dt == ZSAA_BF16) {
      p.N = m->ld_qkv;
      p.pos = m->pos[cur];
      p.cos_t = m->rope_cos;
      p.sin_t = m->rope_sin;
      p.rope_cols = m->dq + m->dkv;
      p.hd = hd;
      p.vnorm_out = m->vnorm;
      TcWeights W{LW(m, li, kWq), LW(m, li, kWk), LW(m, li, kWv), m->dq, m->dq + m->dkv};
      TRACE("gemm_qkv_rope", 2.0 * Md * m->ld_qkv * d, (Md * d + static_cast<double>(m->ld_qkv) * d + Md * m->ld_qkv) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiRope, p, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    } else {
      TRACE("gemm_qkv_f32", 2.0 * Md * m->ld_qkv * d, (Md * d + static_cast<double>(m->ld_qkv) * d + Md * m->ld_qkv) * es);
      trace_scope_.kernels = 1;  // the RoPE kernel below; the GEMMs add theirs
      const int cols[3] = {m->dq, m->dkv, m->dkv};
      const int slots[3] = {kWq, kWk, kWv};
      int c0 = 0;
      for (int t = 0; t < 3; ++t) {
        GemmParams q = p;
        q.N = cols[t];
        q.out = static_cast<float*>(m->qkv) + c0;
        TcWeights W{LW(m, li, slots[t]), nullptr, nullptr, cols[t], cols[t]};
        st = linear(m, m->x, d, W, kEpiStore, q, s, &trace_scope_.kernels);
        if (st != ZSAA_OK) return st;
        c0 += cols[t];
      }
      ZCK(launch_rope_f32(static_cast<float*>(m->qkv), M, m->ld_qkv, m->dq + m->dkv, hd,
                          m->pos[cur], m->rope_cos, m->rope_sin, s));
    }
    if (kc != nullptr) {
      TRACE("kv_write", 0.0, 4.0 * Md * m->dkv * es);
      ZCK(launch_kv_write(m->qkv, m->ld_qkv, m->pos[cur], B, N, Hq, Hkv, hd, kc->layers[li], s));
    }
    {
      const double pairs = static_cast<double>(B) * Hq * n_pairs(N);
      TRACE("attention", 4.0 * pairs * hd, Md * (m->ld_qkv + m->dq) * es + static_cast<double>(B) * Hq * N * 4.0);
      if (attention_pp_supported(dt, hd, Hq, Hkv, nullptr, nullptr, m->status)) {
        ZCK(launch_attention_pp(m->qkv, B, N, Hq, Hkv, hd, m->attn, m->lse, causal, m->status, s));
      } else if (attention_tc_supported(dt, hd, nullptr, nullptr, m->status, m->vt) && attention_tc_preferred(N)) {
        trace_scope_.kernels = 2;  // V transpose + attention
        ZCK(launch_attention_tc(m->qkv, m->vt, B, N, Hq, Hkv, hd, m->attn, m->lse, causal, m->status, s));
      } else {
        ZCK(launch_attention(dt, m->qkv, B, N, Hq, Hkv, hd, m->attn, m->lse, causal, s));
      }
    }
    // A pruning layer's column mass and selection need only q, k and the row
    // normalisers, so its O-projection runs beside them on the side stream;
    // the gather, which reads the updated rows, joins it.  (Not while tracing,
    // which times each launch on the one stream.)
    const bool fork = !m->tracing && prunes(c, l) && sched[l] < N;
    cudaStream_t so = s;
    if (fork) {
      ZCK(fork_side(m, s));
      so = m->side;
    }
    {
      GemmParams q{};
      q.M = M;
      q.N = d;
      q.K = m->dq;
      q.out = h;
      q.ldo = d;
      q.resid = h;
      TcWeights W{LW(m, li, kWo), nullptr, nullptr, d, d};
      TRACE("gemm_o_resid", 2.0 * Md * d * m->dq, (Md * m->dq + static_cast<double>(d) * m->dq + 2.0 * Md * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->attn, m->dq, W, kEpiResid, q, so, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    if (fork) ZCK(cudaEventRecord(m->ev_join, so));
    // Elimination (Sec. 3.3), between attention and MLP: the scores come from
    // this layer's attention and the MLP acts on each row alone, so the kept
    // rows come out exactly as if the whole layer ran first -- but the MLP
    // only runs on the kept rows.
    bool mlp_x_ready = false;
    if (prunes(c, l)) {
      const int k = sched[l];
      const bool want_scores = opts && opts->scores_out;
      const bool forced = opts && opts->forced_idx;
      const bool want_idx = opts && opts->idx_out;
      if (k < N || want_scores || want_idx) {
        float* sc = want_scores ? opts->scores_out + off_scores : m->scores;
        const double pairs = static_cast<double>(B) * Hq * n_pairs(N);
        const int32_t* idx = m->idx;
        if (dt == ZSAA_BF16 && !forced && k < N && N <= kSelectPartsMaxN) {
          // column-mass partials, then top-k with the score reduction fused in
          int n_qc = 1;
          {
            TRACE("colmass", 2.0 * pairs * hd,
                  Md * (m->dq + 2 * m->dkv) * es + static_cast<double>(B) * Hq * N * 4.0);
            ZCK(launch_position_parts(dt, m->qkv, m->lse, dt == ZSAA_BF16 ? m->vnorm : nullptr, B, N,
                                      Hq, Hkv, hd, c.score_mode, m->colmass, &n_qc, m->status,
                                      causal, s));
          }
          TRACE("select", 0.0, static_cast<double>(n_qc) * B * Hkv * N * 4.0 + static_cast<double>(B) * k * 4.0);
          ZCK(launch_select_parts(m->colmass, n_qc, B, Hkv, N, k, c.force_keep_last, m->idx,
                                  want_scores ? sc : nullptr, s));
        } else {
          {
            TRACE("colmass", 2.0 * pairs * hd,
                  Md * (m->dq + 2 * m->dkv) * es + static_cast<double>(B) * Hq * N * 4.0 + Md * 4.0);
            trace_scope_.kernels = 2;
            ZCK(launch_position_scores(dt, m->qkv, m->lse, dt == ZSAA_BF16 ? m->vnorm : nullptr, B, N,
                                       Hq, Hkv, hd, c.score_mode, m->colmass, sc, m->status,
                                       causal, s));
          }
          if (forced) {
            idx = opts->forced_idx + off_forced;
          } else {  // with k == N (only when idx_out is requested) this yields 0..N-1
            TRACE("select", 0.0, Md * 4.0 + static_cast<double>(B) * k * 4.0);
            ZCK(launch_select(sc, B, N, k, c.force_keep_last, m->idx, s));
          }
        }
        if (want_idx)
          ZCK(cudaMemcpyAsync(opts->idx_out + off_idx, idx, sizeof(int32_t) * B * k,
                              cudaMemcpyDeviceToDevice, s));
        if (k < N) {
          if (fork) ZCK(cudaStreamWaitEvent(s, m->ev_join, 0));  // the O-projection has updated h
          if (fuse_norm) {  // the kept rows and their pre-MLP RMSNorm in one pass
            TRACE("gather_norm", 0.0, static_cast<double>(B) * k * (3.0 * d * es + 12.0));
            ZCK(launch_rows_norm(h, nullptr, 0, 0, idx, N, k, m->pos[cur], B * k, d,
                                 LW(m, li, kMlpNorm), c.rms_eps, m->h[cur ^ 1], m->x,
                                 m->pos[cur ^ 1], m->status, s));
            mlp_x_ready = true;
          } else {
            TRACE("gather", 0.0, static_cast<double>(B) * k * (2.0 * d * es + 12.0));
            ZCK(launch_gather(h, B, N, k, static_cast<int>(d * m->esz), idx, m->h[cur ^ 1],
                              m->pos[cur], m->pos[cur ^ 1], m->status, s));
          }
          cur ^= 1;
        }
      }
      off_forced += static_cast<size_t>(B) * k;
      off_idx += static_cast<size_t>(B) * k;
      off_scores += static_cast<size_t>(B) * N;
      N = k;
    }
    // MLP branch on the rows left after the elimination
    const int Mm = B * N;
    const double Mmd = static_cast<double>(Mm);
    void* hm = m->h[cur];
    if (!mlp_x_ready) {
      TRACE("rmsnorm", 0.0, 2.0 * Mmd * d * es);
      ZCK(launch_rmsnorm(dt, hm, LW(m, li, kMlpNorm), Mm, d, c.rms_eps, m->x, s));
    }
    {
      GemmParams q{};
      q.M = Mm;
      q.N = c.ffn_dim;
      q.K = d;
      q.out = m->act;
      q.ldo = c.ffn_dim;
      TcWeights W{LW(m, li, kWg), LW(m, li, kWu), nullptr, c.ffn_dim, c.ffn_dim};
      const double F = c.ffn_dim;
      TRACE("gemm_gate_up_swiglu", 4.0 * Mmd * F * d, (Mmd * d + 2.0 * F * d + Mmd * F) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiSwiGLU, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      GemmParams q{};
      q.M = Mm;
      q.N = d;
      q.K = c.ffn_dim;
      q.out = hm;
      q.ldo = d;
      q.resid = hm;
      TcWeights W{LW(m, li, kWd), nullptr, nullptr, d, d};
      const double F = c.ffn_dim;
      TRACE("gemm_down_resid", 2.0 * Mmd * d * F, (Mmd * F + F * d + 2.0 * Mmd * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->act, c.ffn_dim, W, kEpiResid, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    x_ready = false;  // the next layer normalises its own input
  }
  // head
  const int M = B * N;
  if (opts && opts->hidden_out)
    ZCK(cudaMemcpyAsync(opts->hidden_out, m->h[cur], M * d * m->esz, cudaMemcpyDeviceToDevice, s));
  if (kc != nullptr) {  // next-token logits: final norm and LM head of the last kept row
    if (fuse_norm) {
      TRACE("gather_norm", 0.0, static_cast<double>(B) * (3.0 * d * es + 12.0));
      ZCK(launch_rows_norm(m->h[cur], nullptr, 0, 0, kc->last_idx, N, 1, m->pos[cur], B, d,
                           m->final_norm, c.rms_eps, m->h[cur ^ 1], m->x, m->pos[cur ^ 1],
                           m->status, s));
    } else {
      {
        TRACE("gather", 0.0, static_cast<double>(B) * (2.0 * d * es + 12.0));
        ZCK(launch_gather(m->h[cur], B, N, 1, static_cast<int>(d * m->esz), kc->last_idx,
                          m->h[cur ^ 1], m->pos[cur], m->pos[cur ^ 1], m->status, s));
      }
      TRACE("rmsnorm", 0.0, 2.0 * static_cast<double>(B) * d * es);
      ZCK(launch_rmsnorm(dt, m->h[cur ^ 1], m->final_norm, B, d, c.rms_eps, m->x, s));
    }
    GemmParams q{};
    q.M = B;
    q.N = c.vocab;
    q.K = d;
    q.out = logits;
    q.ldo = c.vocab;
    TcWeights W{m->head, nullptr, nullptr, c.vocab, c.vocab};
    const double V = c.vocab, Mh = B;
    TRACE("gemm_lm_head", 2.0 * Mh * V * d, (Mh * d + V * d) * es + Mh * V * 4.0);
    trace_scope_.kernels = 0;
    st = linear(m, m->x, d, W, kEpiStoreF32, q, s, &trace_scope_.kernels);
    if (st != ZSAA_OK) return st;
  } else if (c.n_classes > 0) {
    TRACE("cls_head", 2.0 * B * d * c.n_classes, (static_cast<double>(B) * d + static_cast<double>(c.n_classes) * d) * es);
    ZCK(launch_cls_head(dt, m->h[cur], B, N, d, m->final_norm, c.rms_eps, m->head, c.n_classes,
                        logits, s));
  } else {
    {
      TRACE("rmsnorm", 0.0, 2.0 * static_cast<double>(M) * d * es);
      ZCK(launch_rmsnorm(dt, m->h[cur], m->final_norm, M, d, c.rms_eps, m->x, s));
    }
    // With a pinned host destination (and not tracing) the head runs as
    // kHeadSlabs column slabs; the side stream copies each slab to the host
    // while the next one computes, and s joins the copies.
    const bool slabs = m->host_logits != nullptr && !m->tracing && dt == ZSAA_BF16;
    const int n_slabs = slabs ? kHeadSlabs : 1;
    const double V = c.vocab, Mh = M;
    for (int sl = 0; sl < n_slabs; ++sl) {
      const int c0 = slab_col(c.vocab, sl, n_slabs), c1 = slab_col(c.vocab, sl + 1, n_slabs);
      if (c1 <= c0) continue;  // a small vocabulary leaves some slabs empty
      GemmParams q{};
      q.M = M;
      q.N = c1 - c0;
      q.K = d;
      q.out = logits + c0;
      q.ldo = c.vocab;
      const void* w0 = static_cast<const uint8_t*>(m->head) + static_cast<size_t>(c0) * d * m->esz;
      TcWeights W{w0, nullptr, nullptr, c1 - c0, c1 - c0};
      TRACE("gemm_lm_head", 2.0 * Mh * (c1 - c0) * d, (Mh * d + (c1 - c0) * static_cast<double>(d)) * es + Mh * (c1 - c0) * 4.0);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, dt == ZSAA_BF16 ? kEpiStoreF32 : kEpiStore, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
      if (slabs) {
        ZCK(fork_side(m, s));
        ZCK(cudaMemcpy2DAsync(m->host_logits + c0, sizeof(float) * c.vocab, logits + c0,
                              sizeof(float) * c.vocab, sizeof(float) * (c1 - c0), M,
                              cudaMemcpyDeviceToHost, m->side));
      }
    }
    if (slabs) {
      ZCK(cudaEventRecord(m->ev_join, m->side));
      ZCK(cudaStreamWaitEvent(s, m->ev_join, 0));
    }
  }
  if (kept_pos)
    ZCK(cudaMemcpyAsync(kept_pos, m->pos[cur], sizeof(int32_t) * M, cudaMemcpyDeviceToDevice, s));
#undef TRACE
  return ZSAA_OK;
}

// Appendix B's formulation as an inference mode: rows are marked instead of
// removed.  Every layer runs on all B*L rows; a marked row is hidden as a key
// from the layer after its marking on, its query adds nothing to later column
// masses, and only unmarked rows compete at a selection.  The kept rows'
// outputs equal those of the compacted forward; the cost is that of accel 1.
// With reactivate (Appendix B's figure, reading R18) nothing is hidden: every
// layer is the unpruned one, and each pruning layer marks the top N_l of all L
// rows by its own scores, whatever the earlier marks.
zsaa_status run_forward_masked(zsaa_model* m, const int32_t* tok, int B, int L, double accel,
                               float* logits, int32_t* kept_pos, const zsaa_forward_opts* opts,
                               cudaStream_t s, bool reactivate = false) {
  const zsaa_config& c = m->cfg;
  const int d = c.d_model, hd = c.head_dim, Hq = c.n_heads, Hkv = c.n_kv_heads, n = c.n_layers;
  if (c.dtype != ZSAA_BF16 || d % 8 != 0 || d > kRowsNormMaxD)
    return fail(ZSAA_ERR_UNSUPPORTED, "the masked mode needs a bf16 model with d_model <= %d", kRowsNormMaxD);
  if (tok == nullptr || logits == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null token or logits pointer");
  if (B < 1 || B > m->max_B || L < 1 || L > m->max_L)
    return fail(ZSAA_ERR_INVALID_ARG, "B=%d L=%d outside [1,%d] x [1,%d]", B, L, m->max_B, m->max_L);
  if (L > kSelectPartsMaxN) return fail(ZSAA_ERR_UNSUPPORTED, "the masked mode needs L <= %d", kSelectPartsMaxN);
  if (opts && (opts->hidden_out || opts->n_layers_run || opts->hidden_in || opts->pos_in ||
               opts->first_layer || opts->plan_L))
    return fail(ZSAA_ERR_INVALID_ARG, "the masked mode takes only the forced_idx/scores_out/idx_out hooks");
  std::vector<int> sched(n + 1);
  double alpha = 1.0;
  zsaa_status st = plan_impl(c, L, accel, sched.data(), &alpha);
  if (st != ZSAA_OK) return st;
  if (m->alive == nullptr)
    ZCK(cudaMalloc(reinterpret_cast<void**>(&m->alive), static_cast<size_t>(m->max_B) * m->max_L));
  ZCK(cudaMemsetAsync(m->alive, 1, static_cast<size_t>(B) * L, s));
  const int dt = c.dtype;
  const int causal = c.bidirectional ? 0 : 1;
  const double es = static_cast<double>(m->esz);
  const int M = B * L;
  const double Md = static_cast<double>(M);
  void* h = m->h[0];
#define TRACE(name, fl, by) TraceScope trace_scope_(m, name, fl, by, s)
  {
    TRACE("embed_norm", 0.0, Md * (3.0 * d * es + 8.0));
    ZCK(launch_rows_norm(m->embed, tok, c.vocab, L, nullptr, 0, 0, nullptr, M, d,
                         LW(m, 0, kAttnNorm), c.rms_eps, h, m->x, m->pos[0], m->status, s));
  }
  const int32_t* kept = nullptr;  // positions of the unmarked rows after the last selection
  size_t off_forced = 0, off_scores = 0, off_idx = 0;
  const double pairs = static_cast<double>(B) * Hq * (causal ? L * (L + 1.0) / 2.0 : 1.0 * L * L);
  for (int l = 1; l <= n; ++l) {
    const int li = l - 1;
    if (l > 1) {
      TRACE("rmsnorm", 0.0, 2.0 * Md * d * es);
      ZCK(launch_rmsnorm(dt, h, LW(m, li, kAttnNorm), M, d, c.rms_eps, m->x, s));
    }
    {
      GemmParams p{};
      p.M = M;
      p.N = m->ld_qkv;
      p.K = d;
      p.out = m->qkv;
      p.ldo = m->ld_qkv;
      p.pos = m->pos[0];
      p.cos_t = m->rope_cos;
      p.sin_t = m->rope_sin;
      p.rope_cols = m->dq + m->dkv;
      p.hd = hd;
      p.vnorm_out = m->vnorm;
      TcWeights W{LW(m, li, kWq), LW(m, li, kWk), LW(m, li, kWv), m->dq, m->dq + m->dkv};
      TRACE("gemm_qkv_rope", 2.0 * Md * m->ld_qkv * d, (Md * d + static_cast<double>(m->ld_qkv) * d + Md * m->ld_qkv) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiRope, p, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      TRACE("attention", 4.0 * pairs * hd, Md * (m->ld_qkv + m->dq) * es + static_cast<double>(B) * Hq * L * 4.0);
      ZCK(launch_attention(dt, m->qkv, B, L, Hq, Hkv, hd, m->attn, m->lse, causal, s, nullptr,
                           reactivate ? nullptr : m->alive));
    }
    // O-projection beside the column mass and selection (see run_forward);
    // the MLP's RMSNorm joins it
    const bool fork = !m->tracing && prunes(c, l);
    cudaStream_t so = s;
    if (fork) {
      ZCK(fork_side(m, s));
      so = m->side;
    }
    {
      GemmParams q{};
      q.M = M;
      q.N = d;
      q.K = m->dq;
      q.out = h;
      q.ldo = d;
      q.resid = h;
      TcWeights W{LW(m, li, kWo), nullptr, nullptr, d, d};
      TRACE("gemm_o_resid", 2.0 * Md * d * m->dq, (Md * m->dq + static_cast<double>(d) * m->dq + 2.0 * Md * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->attn, m->dq, W, kEpiResid, q, so, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    if (fork) ZCK(cudaEventRecord(m->ev_join, so));
    if (prunes(c, l)) {
      const int k = sched[l];
      const bool want_scores = opts && opts->scores_out;
      const bool forced = opts && opts->forced_idx;
      const bool want_idx = opts && opts->idx_out;
      if ((reactivate ? k < L : k < sched[l - 1]) || want_scores || want_idx) {
        int n_qc = 1;
        {
          TRACE("colmass", 2.0 * pairs * hd, Md * (m->dq + 2 * m->dkv) * es);
          ZCK(launch_position_parts(dt, m->qkv, m->lse, m->vnorm, B, L, Hq, Hkv, hd, c.score_mode,
                                    m->colmass, &n_qc, m->status, causal, s, nullptr, 0,
                                    reactivate ? nullptr : m->alive));
        }
        {
          TRACE("select", 0.0, static_cast<double>(n_qc) * B * Hkv * L * 4.0 + static_cast<double>(B) * k * 4.0);
          ZCK(launch_select_parts(m->colmass, n_qc, B, Hkv, L, k, c.force_keep_last, m->idx,
                                  want_scores ? opts->scores_out + off_scores : nullptr, s, nullptr,
                                  nullptr, (forced || reactivate) ? nullptr : m->alive));
        }
        kept = m->idx;
        if (forced) {
          kept = opts->forced_idx + off_forced;
          if (!reactivate) {  // the marks hide rows from later layers
            TRACE("select", 0.0, static_cast<double>(B) * (L + 4.0 * k));
            ZCK(launch_flags_from_idx(kept, B, L, k, m->alive, m->status, s));
          }
        }
        if (want_idx)
          ZCK(cudaMemcpyAsync(opts->idx_out + off_idx, kept, sizeof(int32_t) * B * k,
                              cudaMemcpyDeviceToDevice, s));
      }
      off_forced += static_cast<size_t>(B) * k;
      off_idx += static_cast<size_t>(B) * k;
      off_scores += static_cast<size_t>(B) * L;
    }
    if (fork) ZCK(cudaStreamWaitEvent(s, m->ev_join, 0));  // the O-projection has updated h
    // the MLP of every row, marked or not (the formulation removes nothing)
    {
      TRACE("rmsnorm", 0.0, 2.0 * Md * d * es);
      ZCK(launch_rmsnorm(dt, h, LW(m, li, kMlpNorm), M, d, c.rms_eps, m->x, s));
    }
    const double F = c.ffn_dim;
    {
      GemmParams q{};
      q.M = M;
      q.N = c.ffn_dim;
      q.K = d;
      q.out = m->act;
      q.ldo = c.ffn_dim;
      TcWeights W{LW(m, li, kWg), LW(m, li, kWu), nullptr, c.ffn_dim, c.ffn_dim};
      TRACE("gemm_gate_up_swiglu", 4.0 * Md * F * d, (Md * d + 2.0 * F * d + Md * F) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiSwiGLU, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      GemmParams q{};
      q.M = M;
      q.N = d;
      q.K = c.ffn_dim;
      q.out = h;
      q.ldo = d;
      q.resid = h;
      TcWeights W{LW(m, li, kWd), nullptr, nullptr, d, d};
      TRACE("gemm_down_resid", 2.0 * Md * d * F, (Md * F + F * d + 2.0 * Md * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->act, c.ffn_dim, W, kEpiResid, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
  }
  // the unmarked rows, in order, through the head
  const int nf = sched[n];
  void* hf = h;
  const int32_t* posf = m->pos[0];
  if (kept != nullptr) {
    TRACE("gather_norm", 0.0, static_cast<double>(B) * nf * (3.0 * d * es + 12.0));
    ZCK(launch_rows_norm(h, nullptr, 0, 0, kept, L, nf, m->pos[0], B * nf, d, m->final_norm,
                         c.rms_eps, m->h[1], m->x, m->pos[1], m->status, s));
    hf = m->h[1];
    posf = m->pos[1];
  } else if (c.n_classes == 0) {
    TRACE("rmsnorm", 0.0, 2.0 * static_cast<double>(B) * nf * d * es);
    ZCK(launch_rmsnorm(dt, h, m->final_norm, B * nf, d, c.rms_eps, m->x, s));
  }
  if (c.n_classes > 0) {
    TRACE("cls_head", 2.0 * B * d * c.n_classes, (static_cast<double>(B) * d + static_cast<double>(c.n_classes) * d) * es);
    ZCK(launch_cls_head(dt, hf, B, nf, d, m->final_norm, c.rms_eps, m->head, c.n_classes, logits, s));
  } else {
    GemmParams q{};
    q.M = B * nf;
    q.N = c.vocab;
    q.K = d;
    q.out = logits;
    q.ldo = c.vocab;
    TcWeights W{m->head, nullptr, nullptr, c.vocab, c.vocab};
    const double V = c.vocab, Mh = static_cast<double>(B) * nf;
    TRACE("gemm_lm_head", 2.0 * Mh * V * d, (Mh * d + V * d) * es + Mh * V * 4.0);
    trace_scope_.kernels = 0;
    st = linear(m, m->x, d, W, kEpiStoreF32, q, s, &trace_scope_.kernels);
    if (st != ZSAA_OK) return st;
  }
  if (kept_pos)
    ZCK(cudaMemcpyAsync(kept_pos, posf, sizeof(int32_t) * B * nf, cudaMemcpyDeviceToDevice, s));
#undef TRACE
  return ZSAA_OK;
}

// Pruned prefill of B sequences of different lengths packed back to back
// (sequence b at rows [cu_l[b], cu_l[b+1]) of layer l's buffers).  The dense
// steps (GEMMs, norms) run on all packed rows at once; attention, column mass,
// selection and compaction take the offsets.  bf16 and the fused row path only.
zsaa_status run_forward_varlen(zsaa_model* m, const int32_t* tok, const int32_t* lengths, int B,
                               double accel, float* logits, int32_t* kept_pos,
                               const zsaa_forward_opts* opts, cudaStream_t s) {
  const zsaa_config& c = m->cfg;
  const int d = c.d_model, hd = c.head_dim, Hq = c.n_heads, Hkv = c.n_kv_heads, n = c.n_layers;
  if (c.dtype != ZSAA_BF16 || d % 8 != 0 || d > kRowsNormMaxD)
    return fail(ZSAA_ERR_UNSUPPORTED, "variable-length batches need a bf16 model with d_model <= %d", kRowsNormMaxD);
  if (tok == nullptr || logits == nullptr || lengths == nullptr)
    return fail(ZSAA_ERR_INVALID_ARG, "null token, lengths or logits pointer");
  if (B < 1 || B > m->max_B) return fail(ZSAA_ERR_INVALID_ARG, "B=%d outside [1,%d]", B, m->max_B);
  if (opts && (opts->hidden_out || opts->n_layers_run || opts->hidden_in || opts->pos_in ||
               opts->first_layer || opts->plan_L))
    return fail(ZSAA_ERR_INVALID_ARG, "variable-length forwards take only the forced_idx/scores_out/idx_out hooks");
  long long T0 = 0;
  for (int b = 0; b < B; ++b) {
    if (lengths[b] < 1 || lengths[b] > m->max_L)
      return fail(ZSAA_ERR_INVALID_ARG, "length %d of sequence %d outside [1,%d]", lengths[b], b, m->max_L);
    T0 += lengths[b];
  }
  if (T0 > static_cast<long long>(m->max_B) * m->max_L)
    return fail(ZSAA_ERR_INVALID_ARG, "%lld packed rows exceed max_B*max_L", T0);
  const int n1 = n + 1;
  std::vector<int> sched(static_cast<size_t>(B) * n1);
  double alpha = 1.0;
  zsaa_status st = plan_varlen_impl(c, lengths, B, accel, sched.data(), &alpha);
  if (st != ZSAA_OK) return st;
  // row offsets per layer boundary, the longest sequence, and the row counts
  std::vector<int> rows(n1), nmax(n1, 0);
  if (m->vl_cu == nullptr) {
    ZCK(cudaMalloc(reinterpret_cast<void**>(&m->vl_cu), sizeof(int32_t) * n1 * (m->max_B + 1)));
    ZCK(cudaMallocHost(reinterpret_cast<void**>(&m->vl_cu_host), sizeof(int32_t) * n1 * (m->max_B + 1)));
    ZCK(cudaEventCreateWithFlags(&m->vl_done, cudaEventDisableTiming));
  } else {
    ZCK(cudaEventSynchronize(m->vl_done));  // the previous call's upload has read the host copy
  }
  for (int l = 0; l < n1; ++l) {
    int32_t* cu = m->vl_cu_host + static_cast<size_t>(l) * (B + 1);
    cu[0] = 0;
    for (int b = 0; b < B; ++b) {
      const int nb = sched[static_cast<size_t>(b) * n1 + l];
      cu[b + 1] = cu[b] + nb;
      nmax[l] = nb > nmax[l] ? nb : nmax[l];
    }
    rows[l] = cu[B];
  }
  ZCK(cudaMemcpyAsync(m->vl_cu, m->vl_cu_host, sizeof(int32_t) * n1 * (B + 1), cudaMemcpyHostToDevice, s));
  ZCK(cudaEventRecord(m->vl_done, s));
  auto cu_dev = [&](int l) { return m->vl_cu + static_cast<size_t>(l) * (B + 1); };

  const int dt = c.dtype;
  const int causal = c.bidirectional ? 0 : 1;
  const double es = static_cast<double>(m->esz);
  int cur = 0;
#define TRACE(name, fl, by) TraceScope trace_scope_(m, name, fl, by, s)
  {
    TRACE("embed_norm", 0.0, static_cast<double>(T0) * (3.0 * d * es + 8.0));
    ZCK(launch_rows_norm(m->embed, tok, c.vocab, 1, nullptr, 0, 0, nullptr, rows[0], d,
                         LW(m, 0, kAttnNorm), c.rms_eps, m->h[cur], m->x, m->pos[cur], m->status,
                         s, nullptr, cu_dev(0), B));
  }
  bool x_ready = true;
  size_t off_forced = 0, off_scores = 0, off_idx = 0;
  for (int l = 1; l <= n; ++l) {
    const int li = l - 1;
    const int M = rows[li], Nm = nmax[li];
    const double Md = static_cast<double>(M);
    void* h = m->h[cur];
    if (!x_ready) {
      TRACE("rmsnorm", 0.0, 2.0 * Md * d * es);
      ZCK(launch_rmsnorm(dt, h, LW(m, li, kAttnNorm), M, d, c.rms_eps, m->x, s));
    }
    {
      GemmParams p{};
      p.M = M;
      p.N = m->ld_qkv;
      p.K = d;
      p.out = m->qkv;
      p.ldo = m->ld_qkv;
      p.pos = m->pos[cur];
      p.cos_t = m->rope_cos;
      p.sin_t = m->rope_sin;
      p.rope_cols = m->dq + m->dkv;
      p.hd = hd;
      p.vnorm_out = m->vnorm;
      TcWeights W{LW(m, li, kWq), LW(m, li, kWk), LW(m, li, kWv), m->dq, m->dq + m->dkv};
      TRACE("gemm_qkv_rope", 2.0 * Md * m->ld_qkv * d, (Md * d + static_cast<double>(m->ld_qkv) * d + Md * m->ld_qkv) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiRope, p, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      double pairs = 0.0;
      for (int b = 0; b < B; ++b) {
        const double nb = sched[static_cast<size_t>(b) * n1 + li];
        pairs += causal ? nb * (nb + 1) / 2.0 : nb * nb;
      }
      TRACE("attention", 4.0 * pairs * Hq * hd, Md * (m->ld_qkv + m->dq) * es + static_cast<double>(B) * Hq * Nm * 4.0);
      ZCK(launch_attention(dt, m->qkv, B, Nm, Hq, Hkv, hd, m->attn, m->lse, causal, s, cu_dev(li)));
    }
    // O-projection beside the column mass and selection (see run_forward)
    const bool fork = !m->tracing && prunes(c, l) && rows[l] < M && Nm <= kSelectPartsMaxN;
    cudaStream_t so = s;
    if (fork) {
      ZCK(fork_side(m, s));
      so = m->side;
    }
    {
      GemmParams q{};
      q.M = M;
      q.N = d;
      q.K = m->dq;
      q.out = h;
      q.ldo = d;
      q.resid = h;
      TcWeights W{LW(m, li, kWo), nullptr, nullptr, d, d};
      TRACE("gemm_o_resid", 2.0 * Md * d * m->dq, (Md * m->dq + static_cast<double>(d) * m->dq + 2.0 * Md * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->attn, m->dq, W, kEpiResid, q, so, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    if (fork) ZCK(cudaEventRecord(m->ev_join, so));
    // elimination between attention and MLP (see run_forward), per sequence
    bool mlp_x_ready = false;
    if (prunes(c, l)) {
      const bool want_scores = opts && opts->scores_out;
      const bool forced = opts && opts->forced_idx;
      const bool want_idx = opts && opts->idx_out;
      const bool shrinks = rows[l] < M;
      if (shrinks || want_scores || want_idx) {
        if (Nm > kSelectPartsMaxN)
          return fail(ZSAA_ERR_UNSUPPORTED, "variable-length selection needs lengths <= %d", kSelectPartsMaxN);
        int n_qc = 1;
        {
          TRACE("colmass", 2.0 * Md * Nm * Hq * hd, Md * (m->dq + 2 * m->dkv) * es);
          ZCK(launch_position_parts(dt, m->qkv, m->lse, m->vnorm, B, Nm, Hq, Hkv, hd, c.score_mode,
                                    m->colmass, &n_qc, m->status, causal, s, cu_dev(li), M));
        }
        {
          TRACE("select", 0.0, static_cast<double>(n_qc) * B * Hkv * Nm * 4.0 + rows[l] * 4.0);
          ZCK(launch_select_parts(m->colmass, n_qc, B, Hkv, Nm, 0, c.force_keep_last, m->idx,
                                  want_scores ? opts->scores_out + off_scores : nullptr, s, cu_dev(li),
                                  cu_dev(l)));
        }
        const int32_t* idx = forced ? opts->forced_idx + off_forced : m->idx;
        if (want_idx)
          ZCK(cudaMemcpyAsync(opts->idx_out + off_idx, idx, sizeof(int32_t) * rows[l],
                              cudaMemcpyDeviceToDevice, s));
        if (shrinks) {
          if (fork) ZCK(cudaStreamWaitEvent(s, m->ev_join, 0));  // the O-projection has updated h
          TRACE("gather_norm", 0.0, static_cast<double>(rows[l]) * (3.0 * d * es + 12.0));
          ZCK(launch_rows_norm(h, nullptr, 0, 0, idx, Nm, 0, m->pos[cur], rows[l], d,
                               LW(m, li, kMlpNorm), c.rms_eps, m->h[cur ^ 1], m->x, m->pos[cur ^ 1],
                               m->status, s, cu_dev(li), cu_dev(l), B));
          mlp_x_ready = true;
          cur ^= 1;
        }
      }
      off_forced += rows[l];
      off_idx += rows[l];
      off_scores += M;
    }
    const int Mm = rows[l];
    const double Mmd = static_cast<double>(Mm);
    void* hm = m->h[cur];
    if (!mlp_x_ready) {
      TRACE("rmsnorm", 0.0, 2.0 * Mmd * d * es);
      ZCK(launch_rmsnorm(dt, hm, LW(m, li, kMlpNorm), Mm, d, c.rms_eps, m->x, s));
    }
    const double F = c.ffn_dim;
    {
      GemmParams q{};
      q.M = Mm;
      q.N = c.ffn_dim;
      q.K = d;
      q.out = m->act;
      q.ldo = c.ffn_dim;
      TcWeights W{LW(m, li, kWg), LW(m, li, kWu), nullptr, c.ffn_dim, c.ffn_dim};
      TRACE("gemm_gate_up_swiglu", 4.0 * Mmd * F * d, (Mmd * d + 2.0 * F * d + Mmd * F) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiSwiGLU, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      GemmParams q{};
      q.M = Mm;
      q.N = d;
      q.K = c.ffn_dim;
      q.out = hm;
      q.ldo = d;
      q.resid = hm;
      TcWeights W{LW(m, li, kWd), nullptr, nullptr, d, d};
      TRACE("gemm_down_resid", 2.0 * Mmd * d * F, (Mmd * F + F * d + 2.0 * Mmd * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->act, c.ffn_dim, W, kEpiResid, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    x_ready = false;
  }
  const int Mf = rows[n];
  if (c.n_classes > 0) {
    TRACE("cls_head", 2.0 * B * d * c.n_classes, (static_cast<double>(B) * d + static_cast<double>(c.n_classes) * d) * es);
    ZCK(launch_cls_head(dt, m->h[cur], B, 0, d, m->final_norm, c.rms_eps, m->head, c.n_classes,
                        logits, s, cu_dev(n)));
  } else {
    {
      TRACE("rmsnorm", 0.0, 2.0 * static_cast<double>(Mf) * d * es);
      ZCK(launch_rmsnorm(dt, m->h[cur], m->final_norm, Mf, d, c.rms_eps, m->x, s));
    }
    GemmParams q{};
    q.M = Mf;
    q.N = c.vocab;
    q.K = d;
    q.out = logits;
    q.ldo = c.vocab;
    TcWeights W{m->head, nullptr, nullptr, c.vocab, c.vocab};
    const double V = c.vocab, Mh = Mf;
    TRACE("gemm_lm_head", 2.0 * Mh * V * d, (Mh * d + V * d) * es + Mh * V * 4.0);
    trace_scope_.kernels = 0;
    st = linear(m, m->x, d, W, kEpiStoreF32, q, s, &trace_scope_.kernels);
    if (st != ZSAA_OK) return st;
  }
  if (kept_pos)
    ZCK(cudaMemcpyAsync(kept_pos, m->pos[cur], sizeof(int32_t) * Mf, cudaMemcpyDeviceToDevice, s));
#undef TRACE
  return ZSAA_OK;
}

// A plain forward (no hooks, not tracing) is replayed from a CUDA graph: the
// first call with given arguments runs eagerly, the second is captured and
// instantiated, later ones launch the graph (one launch instead of ~175 and
// no per-call host work).  At most kMaxGraphs argument sets are kept.
constexpr size_t kMaxGraphs = 16;

zsaa_status forward_cached(zsaa_model* m, const int32_t* tok, int B, int L, double accel,
                           float* logits, int32_t* kept_pos, cudaStream_t s,
                           zsaa_cache* kc = nullptr) {
  if (!m->use_graphs || m->tracing)
    return run_forward(m, tok, B, L, accel, logits, kept_pos, nullptr, s, kc);
  char key[200];
  snprintf(key, sizeof(key), "%p/%d/%d/%.17g/%p/%p/%p/%p", static_cast<const void*>(tok), B, L, accel,
           static_cast<void*>(logits), static_cast<void*>(kept_pos), static_cast<void*>(kc),
           static_cast<void*>(m->host_logits));
  auto it = m->graphs.begin();
  for (; it != m->graphs.end(); ++it)
    if (it->key == key) break;
  if (it == m->graphs.end()) {
    m->graphs.push_front(zsaa_model::GraphEntry{key, 0, nullptr, kc});
    if (m->graphs.size() > kMaxGraphs) {
      if (m->graphs.back().exec) cudaGraphExecDestroy(m->graphs.back().exec);
      m->graphs.pop_back();
    }
    it = m->graphs.begin();
  } else if (it != m->graphs.begin()) {
    m->graphs.splice(m->graphs.begin(), m->graphs, it);
    it = m->graphs.begin();
  }
  if (it->exec != nullptr) {
    ZCK(cudaGraphLaunch(it->exec, s));
    return ZSAA_OK;
  }
  if (it->seen == 0) {  // first sight: eager (also sets up kernel attributes)
    zsaa_status st = run_forward(m, tok, B, L, accel, logits, kept_pos, nullptr, s, kc);
    if (st == ZSAA_OK) it->seen = 1;
    return st;
  }
  // Record on the model's own stream (capture is impossible on the legacy
  // default stream); recording executes nothing, the launch below does.
  if (m->capture_stream == nullptr)
    ZCK(cudaStreamCreateWithFlags(&m->capture_stream, cudaStreamNonBlocking));
  cudaGraph_t graph = nullptr;
  ZCK(cudaStreamBeginCapture(m->capture_stream, cudaStreamCaptureModeThreadLocal));
  zsaa_status st = run_forward(m, tok, B, L, accel, logits, kept_pos, nullptr, m->capture_stream, kc);
  cudaError_t e = cudaStreamEndCapture(m->capture_stream, &graph);
  if (st != ZSAA_OK) {
    if (graph) cudaGraphDestroy(graph);
    return st;
  }
  ZCK(e);
  cudaGraphExec_t exec = nullptr;
  e = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  ZCK(e);
  it->exec = exec;
  ZCK(cudaGraphLaunch(exec, s));
  return ZSAA_OK;
}

zsaa_status score_select_impl(const void* hidden, int B, int L, int d, int dtype, int k, int flags,
                              const float* scores_in, float* scores_out, int32_t* idx_out,
                              void* gathered_out, cudaStream_t s) {
  if (hidden == nullptr || idx_out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null hidden or idx_out");
  if (B < 1 || L < 1 || d < 1) return fail(ZSAA_ERR_INVALID_ARG, "B, L, d must be >= 1");
  if (k < 1 || k > L) return fail(ZSAA_ERR_INVALID_ARG, "k=%d outside [1, L=%d]", k, L);
  if (dtype != ZSAA_BF16 && dtype != ZSAA_F32) return fail(ZSAA_ERR_INVALID_ARG, "bad dtype");
  const int esz = dtype == ZSAA_BF16 ? 2 : 4;
  if ((static_cast<size_t>(d) * esz) % 16 != 0)
    return fail(ZSAA_ERR_INVALID_ARG, "row bytes d*%d must be a multiple of 16", esz);
  if ((reinterpret_cast<uintptr_t>(hidden) | reinterpret_cast<uintptr_t>(gathered_out)) % 16)
    return fail(ZSAA_ERR_INVALID_ARG, "hidden and gathered_out must be 16-byte aligned");
  if (static_cast<long long>(B) * L > (1LL << 31) - 1)
    return fail(ZSAA_ERR_INVALID_ARG, "B*L too large");
  const int force_last = (flags & ZSAA_FLAG_FORCE_KEEP_LAST) ? 1 : 0;
  float* scratch = nullptr;
  const float* sc = scores_in;
  if (sc == nullptr) {
    float* dst = scores_out;
    if (dst == nullptr) {
      ZCK(cudaMallocAsync(reinterpret_cast<void**>(&scratch), sizeof(float) * B * L, s));
      dst = scratch;
    }
    ZCK(launch_row_norm(dtype, hidden, B * L, d, dst, s));
    sc = dst;
  } else if (scores_out != nullptr) {
    ZCK(cudaMemcpyAsync(scores_out, scores_in, sizeof(float) * B * L, cudaMemcpyDeviceToDevice, s));
  }
  cudaError_t e = launch_select(sc, B, L, k, force_last, idx_out, s);
  if (e == cudaSuccess && gathered_out != nullptr)
    e = launch_gather(hidden, B, L, k, d * esz, idx_out, gathered_out, nullptr, nullptr, nullptr, s);
  if (scratch) {
    cudaError_t e2 = cudaFreeAsync(scratch, s);
    if (e == cudaSuccess) e = e2;
  }
  ZCK(e);
  return ZSAA_OK;
}

zsaa_status read_status(int* word, cudaStream_t s, bool whole_device) {
  if (whole_device)
    ZCK(cudaDeviceSynchronize());
  else
    ZCK(cudaStreamSynchronize(s));
  int v = 0;
  ZCK(cudaMemcpy(&v, word, sizeof(int), cudaMemcpyDeviceToHost));
  if (v != 0) {
    ZCK(cudaMemset(word, 0, sizeof(int)));
    if (v & kStatusTimeout)
      return fail(ZSAA_ERR_TIMEOUT, "a kernel gave up a bounded wait (status 0x%x)", v);
    return fail(ZSAA_ERR_INVALID_ARG, "a token id or forced index was out of range (status 0x%x)", v);
  }
  return ZSAA_OK;
}

// Self-test of the failure path every pipelined kernel takes: two roles wait,
// with the library's bounded mbarrier wait, for a phase of a barrier whose one
// expected arrival never comes (a producer that stopped).  The first wait to
// run out (kWaitLimitNs) sets the timeout bit of the status word and the CTA's
// stop flag; the other role sees the flag and stops; the kernel returns.  No
// trap, no fault: the context stays usable.
__global__ void wait_timeout_selftest_kernel(int* status) {
  __shared__ uint64_t bar;
  __shared__ int stop;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    stop = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if ((threadIdx.x & 31) == 0) mbar_wait_ab(&bar, 0, status, reinterpret_cast<volatile int*>(&stop));
  __syncthreads();
}

// cos/sin of RoPE for positions [0, n_pos): angle(p, i) = p * theta^(-2i/hd), in double.
void rope_host_table(double theta, int hd, int n_pos, std::vector<float>* cs, std::vector<float>* sn) {
  const int half = hd / 2;
  cs->assign(static_cast<size_t>(n_pos) * half, 0.f);
  sn->assign(cs->size(), 0.f);
  for (int p = 0; p < n_pos; ++p)
    for (int i = 0; i < half; ++i) {
      const double a = static_cast<double>(p) *
                       std::pow(theta, -2.0 * static_cast<double>(i) / static_cast<double>(hd));
      (*cs)[static_cast<size_t>(p) * half + i] = static_cast<float>(std::cos(a));
      (*sn)[static_cast<size_t>(p) * half + i] = static_cast<float>(std::sin(a));
    }
}

void free_cache(zsaa_cache* c) {
  if (c == nullptr) return;
  if (c->graph) cudaGraphExecDestroy(c->graph);
  void* ptrs[] = {c->kv, c->pos, c->rope_cos, c->rope_sin, c->qkv32, c->last_idx, c->step};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  delete c;
}

// One generated token per sequence (B rows through every layer, attention over
// the pruned cache), then the next-token logits; the step counter advances last.
zsaa_status run_decode(zsaa_model* m, zsaa_cache* kc, const int32_t* tok, float* logits,
                       cudaStream_t s) {
  const zsaa_config& c = m->cfg;
  const int B = kc->B, d = c.d_model, hd = c.head_dim, Hq = c.n_heads, Hkv = c.n_kv_heads;
  const double es = static_cast<double>(m->esz), Bd = B;
  void* h = m->h[0];
  zsaa_status st = ZSAA_OK;
#define TRACE(name, fl, by) TraceScope trace_scope_(m, name, fl, by, s)
  {
    TRACE("embed_norm", 0.0, Bd * (3.0 * d * es + 8.0));
    ZCK(launch_rows_norm(m->embed, tok, c.vocab, 1, nullptr, 0, 0, nullptr, B, d,
                         LW(m, 0, kAttnNorm), c.rms_eps, h, m->x, m->pos[0], m->status, s));
  }
  for (int li = 0; li < c.n_layers; ++li) {
    if (li > 0) {
      TRACE("rmsnorm", 0.0, 2.0 * Bd * d * es);
      ZCK(launch_rmsnorm(c.dtype, h, LW(m, li, kAttnNorm), B, d, c.rms_eps, m->x, s));
    }
    {
      GemmParams p{};
      p.M = B;
      p.N = m->ld_qkv;
      p.K = d;
      p.out = kc->qkv32;
      p.ldo = m->ld_qkv;
      TcWeights W{LW(m, li, kWq), LW(m, li, kWk), LW(m, li, kWv), m->dq, m->dq + m->dkv};
      TRACE("gemm_qkv", 2.0 * Bd * m->ld_qkv * d, (Bd * d + static_cast<double>(m->ld_qkv) * d) * es + Bd * m->ld_qkv * 4.0);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiStoreF32, p, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      const zsaa::KvLayer& L = kc->layers[li];
      const double keys = static_cast<double>(L.base) + kc->generated + 1;
      TRACE("decode_attention", 4.0 * Bd * Hq * hd * keys, 2.0 * Bd * Hkv * hd * keys * es + Bd * m->ld_qkv * 4.0);
      ZCK(launch_decode_attention(kc->qkv32, m->ld_qkv, B, Hq, Hkv, hd, L, kc->step, kc->L,
                                  kc->rope_cos, kc->rope_sin, m->attn, s));
    }
    {
      GemmParams q{};
      q.M = B;
      q.N = d;
      q.K = m->dq;
      q.out = h;
      q.ldo = d;
      q.resid = h;
      TcWeights W{LW(m, li, kWo), nullptr, nullptr, d, d};
      TRACE("gemm_o_resid", 2.0 * Bd * d * m->dq, (Bd * m->dq + static_cast<double>(d) * m->dq + 2.0 * Bd * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->attn, m->dq, W, kEpiResid, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      TRACE("rmsnorm", 0.0, 2.0 * Bd * d * es);
      ZCK(launch_rmsnorm(c.dtype, h, LW(m, li, kMlpNorm), B, d, c.rms_eps, m->x, s));
    }
    const double F = c.ffn_dim;
    {
      GemmParams q{};
      q.M = B;
      q.N = c.ffn_dim;
      q.K = d;
      q.out = m->act;
      q.ldo = c.ffn_dim;
      TcWeights W{LW(m, li, kWg), LW(m, li, kWu), nullptr, c.ffn_dim, c.ffn_dim};
      TRACE("gemm_gate_up_swiglu", 4.0 * Bd * F * d, (Bd * d + 2.0 * F * d + Bd * F) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->x, d, W, kEpiSwiGLU, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
    {
      GemmParams q{};
      q.M = B;
      q.N = d;
      q.K = c.ffn_dim;
      q.out = h;
      q.ldo = d;
      q.resid = h;
      TcWeights W{LW(m, li, kWd), nullptr, nullptr, d, d};
      TRACE("gemm_down_resid", 2.0 * Bd * d * F, (Bd * F + F * d + 2.0 * Bd * d) * es);
      trace_scope_.kernels = 0;
      st = linear(m, m->act, c.ffn_dim, W, kEpiResid, q, s, &trace_scope_.kernels);
      if (st != ZSAA_OK) return st;
    }
  }
  {
    TRACE("rmsnorm", 0.0, 2.0 * Bd * d * es);
    ZCK(launch_rmsnorm(c.dtype, h, m->final_norm, B, d, c.rms_eps, m->x, s));
  }
  {
    GemmParams q{};
    q.M = B;
    q.N = c.vocab;
    q.K = d;
    q.out = logits;
    q.ldo = c.vocab;
    TcWeights W{m->head, nullptr, nullptr, c.vocab, c.vocab};
    const double V = c.vocab;
    TRACE("gemm_lm_head", 2.0 * Bd * V * d, (Bd * d + V * d) * es + Bd * V * 4.0);
    trace_scope_.kernels = 0;
    st = linear(m, m->x, d, W, kEpiStoreF32, q, s, &trace_scope_.kernels);
    if (st != ZSAA_OK) return st;
  }
  {
    TRACE("advance", 0.0, 8.0);
    ZCK(launch_decode_advance(kc->step, s));
  }
#undef TRACE
  return ZSAA_OK;
}

// The decode step reads its position from device memory, so one graph serves
// every step: the first call with given pointers runs eagerly, the second is
// recorded, later ones launch the recording.
zsaa_status decode_cached(zsaa_model* m, zsaa_cache* kc, const int32_t* tok, float* logits,
                          cudaStream_t s) {
  if (!m->use_graphs || m->tracing) return run_decode(m, kc, tok, logits, s);
  char key[96];
  snprintf(key, sizeof(key), "%p/%p", static_cast<const void*>(tok), static_cast<void*>(logits));
  if (kc->graph_key != key) {
    if (kc->graph) cudaGraphExecDestroy(kc->graph);
    kc->graph = nullptr;
    kc->graph_key = key;
    kc->graph_seen = 0;
  }
  if (kc->graph) {
    ZCK(cudaGraphLaunch(kc->graph, s));
    return ZSAA_OK;
  }
  if (kc->graph_seen == 0) {
    zsaa_status st = run_decode(m, kc, tok, logits, s);
    if (st == ZSAA_OK) kc->graph_seen = 1;
    return st;
  }
  if (m->capture_stream == nullptr)
    ZCK(cudaStreamCreateWithFlags(&m->capture_stream, cudaStreamNonBlocking));
  cudaGraph_t graph = nullptr;
  ZCK(cudaStreamBeginCapture(m->capture_stream, cudaStreamCaptureModeThreadLocal));
  zsaa_status st = run_decode(m, kc, tok, logits, m->capture_stream);
  cudaError_t e = cudaStreamEndCapture(m->capture_stream, &graph);
  if (st != ZSAA_OK) {
    if (graph) cudaGraphDestroy(graph);
    return st;
  }
  ZCK(e);
  cudaGraphExec_t exec = nullptr;
  e = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  ZCK(e);
  kc->graph = exec;
  ZCK(cudaGraphLaunch(exec, s));
  return ZSAA_OK;
}

}  // namespace

// ================================================================ C ABI

extern "C" {

const char* zsaa_last_error(void) { return g_last_error.c_str(); }

const char* zsaa_version(void) { return "zsaa 0.1 (sm_103a)"; }

zsaa_status zsaa_plan_config(const zsaa_config* cfg, int L, double accel, int* n_sched,
                             double* alpha_out) {
  if (cfg == nullptr || n_sched == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  zsaa_status st = validate_config(*cfg);
  if (st != ZSAA_OK) return st;
  return plan_impl(*cfg, L, accel, n_sched, alpha_out);
}

zsaa_status zsaa_model_create(const zsaa_config* cfg, const zsaa_weights* w, int max_B, int max_L,
                              zsaa_model** out) {
  if (out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null out");
  *out = nullptr;
  if (cfg == nullptr || w == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null config or weights");
  zsaa_status st = validate_config(*cfg);
  if (st != ZSAA_OK) return st;
  if (max_B < 1 || max_L < 1) return fail(ZSAA_ERR_INVALID_ARG, "max_B and max_L must be >= 1");
  if (w->embed == nullptr || w->layers == nullptr || w->final_norm == nullptr || w->head == nullptr)
    return fail(ZSAA_ERR_INVALID_ARG, "null weight pointer");
  const size_t esz = cfg->dtype == ZSAA_BF16 ? 2 : 4;
  for (int i = 0; i < cfg->n_layers * 9; ++i) {
    const void* p = w->layers[i];
    if (p == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null layer weight %d", i);
    if (reinterpret_cast<uintptr_t>(p) % 16) return fail(ZSAA_ERR_INVALID_ARG, "layer weight %d not 16-byte aligned", i);
  }
  const long long rows = static_cast<long long>(max_B) * max_L;
  if (rows > (1LL << 30)) return fail(ZSAA_ERR_INVALID_ARG, "max_B*max_L too large");

  zsaa_model* m = new zsaa_model();
  m->cfg = *cfg;
  m->max_B = max_B;
  m->max_L = max_L;
  cudaGetDevice(&m->device);
  m->embed = w->embed;
  m->final_norm = w->final_norm;
  m->head = w->head;
  m->layers.assign(w->layers, w->layers + cfg->n_layers * 9);
  m->esz = esz;
  m->dq = cfg->n_heads * cfg->head_dim;
  m->dkv = cfg->n_kv_heads * cfg->head_dim;
  m->ld_qkv = m->dq + 2 * m->dkv;

  const size_t d = cfg->d_model, F = cfg->ffn_dim;
  bool ok = true;
  auto alloc = [&](void** p, size_t bytes) {
    if (ok && cudaMalloc(p, bytes + 16) != cudaSuccess) ok = false;
  };
  alloc(&m->h[0], rows * d * esz);
  alloc(&m->h[1], rows * d * esz);
  alloc(&m->x, rows * d * esz);
  alloc(&m->qkv, rows * m->ld_qkv * esz);
  alloc(&m->attn, rows * m->dq * esz);
  alloc(&m->act, rows * F * esz);
  alloc(reinterpret_cast<void**>(&m->lse), rows * cfg->n_heads * sizeof(float));
  if (cfg->dtype == ZSAA_BF16 && (cfg->head_dim == 64 || cfg->head_dim == 128))
    alloc(&m->vt, attention_tc_vt_elems(max_B, max_L, cfg->n_kv_heads, cfg->head_dim) * 2);
  alloc(reinterpret_cast<void**>(&m->colmass),
        colmass_parts_elems(max_B, max_L, cfg->n_heads, cfg->n_kv_heads) * sizeof(float));
  alloc(reinterpret_cast<void**>(&m->vnorm), rows * cfg->n_kv_heads * sizeof(float));
  alloc(reinterpret_cast<void**>(&m->scores), rows * sizeof(float));
  alloc(reinterpret_cast<void**>(&m->idx), rows * sizeof(int32_t));
  alloc(reinterpret_cast<void**>(&m->pos[0]), rows * sizeof(int32_t));
  alloc(reinterpret_cast<void**>(&m->pos[1]), rows * sizeof(int32_t));
  const int half = cfg->head_dim / 2;
  alloc(reinterpret_cast<void**>(&m->rope_cos), static_cast<size_t>(max_L) * half * sizeof(float));
  alloc(reinterpret_cast<void**>(&m->rope_sin), static_cast<size_t>(max_L) * half * sizeof(float));
  alloc(reinterpret_cast<void**>(&m->status), sizeof(int));
  if (cfg->dtype == ZSAA_BF16) {
    alloc(reinterpret_cast<void**>(&m->splitk_ws), kSplitKWorkspaceElems * sizeof(float));
    alloc(reinterpret_cast<void**>(&m->splitk_flags), kSplitKFlags * sizeof(int));
  }
  if (!ok) {
    cudaGetLastError();
    free_model(m);
    return fail(ZSAA_ERR_OOM, "workspace allocation failed for max_B=%d max_L=%d", max_B, max_L);
  }
  // RoPE table: angle(p, i) = p * theta^(-2i/hd), evaluated in double.
  std::vector<float> cs(static_cast<size_t>(max_L) * half), sn(cs.size());
  for (int p = 0; p < max_L; ++p)
    for (int i = 0; i < half; ++i) {
      const double inv = std::pow(static_cast<double>(cfg->rope_theta),
                                  -2.0 * static_cast<double>(i) / static_cast<double>(cfg->head_dim));
      const double a = static_cast<double>(p) * inv;
      cs[static_cast<size_t>(p) * half + i] = static_cast<float>(std::cos(a));
      sn[static_cast<size_t>(p) * half + i] = static_cast<float>(std::sin(a));
    }
  cudaError_t e = cudaMemcpy(m->rope_cos, cs.data(), cs.size() * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(m->rope_sin, sn.data(), sn.size() * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(m->status, 0, sizeof(int));
  if (e == cudaSuccess && m->splitk_flags) e = cudaMemset(m->splitk_flags, 0, kSplitKFlags * sizeof(int));
  if (e != cudaSuccess) {
    free_model(m);
    return fail(ZSAA_ERR_CUDA, "workspace initialisation failed: %s", cudaGetErrorString(e));
  }
  if (cfg->dtype == ZSAA_BF16 && get_encode_tiled() == nullptr) {
    free_model(m);
    return fail(ZSAA_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  }
  *out = m;
  return ZSAA_OK;
}

void zsaa_model_destroy(zsaa_model* m) {
  if (m == nullptr) return;
  cudaDeviceSynchronize();
  free_model(m);
}

zsaa_status zsaa_plan(const zsaa_model* m, int L, double accel, int* n_sched, double* alpha_out) {
  if (m == nullptr || n_sched == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  return plan_impl(m->cfg, L, accel, n_sched, alpha_out);
}

zsaa_status zsaa_forward(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                         float* logits_out, int32_t* kept_pos_out, zsaa_stream stream) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  return forward_cached(m, token_ids, B, L, accel, logits_out, kept_pos_out,
                        reinterpret_cast<cudaStream_t>(stream));
}

zsaa_status zsaa_model_set_graphs(zsaa_model* m, int enable) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  m->use_graphs = enable != 0;
  return ZSAA_OK;
}

zsaa_status zsaa_forward_ex(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                            float* logits_out, int32_t* kept_pos_out, const zsaa_forward_opts* opts,
                            zsaa_stream stream) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  return run_forward(m, token_ids, B, L, accel, logits_out, kept_pos_out, opts,
                     reinterpret_cast<cudaStream_t>(stream));
}

zsaa_status zsaa_forward_host(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                              float* logits_out, int32_t* kept_pos_out, zsaa_stream stream) {
  if (m == nullptr || token_ids == nullptr || logits_out == nullptr)
    return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  if (B < 1 || B > m->max_B || L < 1 || L > m->max_L)
    return fail(ZSAA_ERR_INVALID_ARG, "B=%d L=%d outside [1,%d] x [1,%d]", B, L, m->max_B, m->max_L);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  std::vector<int> sched(m->cfg.n_layers + 1);
  zsaa_status st = plan_impl(m->cfg, L, accel, sched.data(), nullptr);
  if (st != ZSAA_OK) return st;
  const int n_final = sched[m->cfg.n_layers];
  const size_t n_logits = m->cfg.n_classes > 0 ? static_cast<size_t>(B) * m->cfg.n_classes
                                               : static_cast<size_t>(B) * n_final * m->cfg.vocab;
  const size_t rows = static_cast<size_t>(m->max_B) * m->max_L;
  if (m->stage_tok == nullptr) {
    ZCK(cudaMalloc(&m->stage_tok, rows * sizeof(int32_t)));
    ZCK(cudaMalloc(&m->stage_pos, rows * sizeof(int32_t)));
  }
  if (m->stage_logits_cap < n_logits) {
    if (m->stage_logits) ZCK(cudaFree(m->stage_logits));
    m->stage_logits = nullptr;
    m->stage_logits_cap = 0;
    ZCK(cudaMalloc(&m->stage_logits, n_logits * sizeof(float)));
    m->stage_logits_cap = n_logits;
  }
  // A pinned (page-locked) logits buffer lets the LM head's column slabs be
  // copied while later slabs compute; other buffers get one copy at the end.
  bool stream_logits = false;
  if (m->cfg.n_classes == 0 && m->cfg.dtype == ZSAA_BF16) {
    cudaPointerAttributes pa{};
    if (cudaPointerGetAttributes(&pa, logits_out) == cudaSuccess)
      stream_logits = pa.type == cudaMemoryTypeHost;
    else
      cudaGetLastError();
  }
  ZCK(cudaMemcpyAsync(m->stage_tok, token_ids, sizeof(int32_t) * B * L, cudaMemcpyHostToDevice, s));
  m->host_logits = stream_logits ? logits_out : nullptr;
  st = forward_cached(m, m->stage_tok, B, L, accel, m->stage_logits, m->stage_pos, s);
  m->host_logits = nullptr;
  if (st != ZSAA_OK) return st;
  if (!stream_logits)
    ZCK(cudaMemcpyAsync(logits_out, m->stage_logits, n_logits * sizeof(float), cudaMemcpyDeviceToHost, s));
  if (kept_pos_out)
    ZCK(cudaMemcpyAsync(kept_pos_out, m->stage_pos, sizeof(int32_t) * B * n_final,
                        cudaMemcpyDeviceToHost, s));
  ZCK(cudaStreamSynchronize(s));
  return ZSAA_OK;
}

zsaa_status zsaa_score_select(const void* hidden, int B, int L, int d, int k, int32_t* idx_out,
                              void* gathered_out, zsaa_stream stream) {
  return score_select_impl(hidden, B, L, d, ZSAA_BF16, k, 0, nullptr, nullptr, idx_out,
                           gathered_out, reinterpret_cast<cudaStream_t>(stream));
}

zsaa_status zsaa_score_select_ex(const void* hidden, int B, int L, int d, int dtype, int k,
                                 int flags, const float* scores_in, float* scores_out,
                                 int32_t* idx_out, void* gathered_out, zsaa_stream stream) {
  return score_select_impl(hidden, B, L, d, dtype, k, flags, scores_in, scores_out, idx_out,
                           gathered_out, reinterpret_cast<cudaStream_t>(stream));
}

zsaa_status zsaa_gemm_schedule(int epilogue, int M, int N, int K, int hd, int sms, int pair_slots,
                               int split_slots, int32_t* plan_out, int32_t* items, int64_t cap,
                               int64_t* n_items) {
  if (plan_out == nullptr || n_items == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  if (items == nullptr && cap != 0) return fail(ZSAA_ERR_INVALID_ARG, "null items with cap > 0");
  if (cap < 0) return fail(ZSAA_ERR_INVALID_ARG, "cap must be >= 0");
  if (M < 1 || N < 16 || K < 64) return fail(ZSAA_ERR_INVALID_ARG, "M >= 1, N >= 16, K >= 64");
  if (K % 64 || N % 16) return fail(ZSAA_ERR_UNSUPPORTED, "the tiled GEMM needs K %% 64 == 0 and N %% 16 == 0");
  if (epilogue < 0 || epilogue > 4) return fail(ZSAA_ERR_INVALID_ARG, "bad epilogue");
  if (epilogue == kEpiRope && (hd < 32 || hd % 32)) return fail(ZSAA_ERR_INVALID_ARG, "bad RoPE head size");
  if (sms < 1 || pair_slots < 0 || split_slots < 0) return fail(ZSAA_ERR_INVALID_ARG, "bad device description");
  // tile counts are ints: at most 2^31 - 1 tiles of the narrowest plan (128 x 64)
  if ((static_cast<long long>(M) + 127) / 128 * ((2LL * N + 63) / 64) > 0x7fffffffLL)
    return fail(ZSAA_ERR_UNSUPPORTED, "shape too large for the tile plan");
  long long n = 0;
  const int r = gemm_tc_schedule(epilogue, M, N, K, hd, sms, pair_slots, split_slots, plan_out, items, cap, &n);
  if (r == -1) return fail(ZSAA_ERR_UNSUPPORTED, "no tile plan for this shape");
  if (r != 0) return fail(ZSAA_ERR_INVALID_ARG, "work items outnumber the tiles' k-blocks");
  *n_items = n;
  return ZSAA_OK;
}

zsaa_status zsaa_op_linear(const void* A, const void* W, const void* W2, const void* resid,
                           void* out, int M, int N, int K, int dtype, int epilogue,
                           const int32_t* pos, int rope_cols, int rope_hd, float rope_theta,
                           zsaa_stream stream) {
  if (A == nullptr || W == nullptr || out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  if (M < 1 || N < 1 || K < 1) return fail(ZSAA_ERR_INVALID_ARG, "M, N, K must be >= 1");
  if (epilogue < 0 || epilogue > 4) return fail(ZSAA_ERR_INVALID_ARG, "bad epilogue");
  if (epilogue == kEpiSwiGLU && W2 == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "SwiGLU needs W2");
  if (epilogue == kEpiResid && resid == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "residual needs resid");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  GemmParams p{};
  p.M = M;
  p.N = N;
  p.K = K;
  p.out = out;
  p.ldo = N;
  p.resid = resid;
  p.status = shared_status();
  if (p.status == nullptr) return fail(ZSAA_ERR_CUDA, "status word allocation failed");
  if (dtype == ZSAA_BF16) {
    if (K % 64 || N % 16) return fail(ZSAA_ERR_UNSUPPORTED, "bf16 GEMM needs K %% 64 == 0 and N %% 16 == 0");
    if (epilogue == kEpiRope) {
      if (pos == nullptr || rope_hd < 32 || rope_hd % 32 || rope_cols % rope_hd || rope_cols > N)
        return fail(ZSAA_ERR_INVALID_ARG, "bad RoPE arguments");
      RopeTable t;
      if (!op_rope_table(rope_theta, rope_hd, &t)) return fail(ZSAA_ERR_CUDA, "RoPE table setup failed");
      p.pos = pos;
      p.cos_t = t.cos_t;
      p.sin_t = t.sin_t;
      p.rope_cols = rope_cols;
      p.hd = rope_hd;
    }
    TcWeights Wt{W, W2, nullptr, N, N};
    if (!op_splitk_ws(&p.splitk_ws, &p.splitk_flags)) p.splitk_ws = nullptr, p.splitk_flags = nullptr;
    p.splitk_ws_elems = p.splitk_ws ? kSplitKWorkspaceElems : 0;
    ZCK(launch_gemm_tc(A, K, Wt, epilogue, p, s));
  } else if (dtype == ZSAA_F32) {
    if (epilogue == kEpiRope) return fail(ZSAA_ERR_UNSUPPORTED, "f32 GEMM has no RoPE epilogue");
    ZCK(launch_gemm_f32(static_cast<const float*>(A), K, static_cast<const float*>(W),
                        static_cast<const float*>(W2), epilogue, p, s));
  } else {
    return fail(ZSAA_ERR_INVALID_ARG, "bad dtype");
  }
  return ZSAA_OK;
}

zsaa_status zsaa_op_attention(const void* qkv, int B, int N, int Hq, int Hkv, int hd, int dtype,
                              void* out, float* lse, zsaa_stream stream) {
  return zsaa_op_attention_ex(qkv, B, N, Hq, Hkv, hd, dtype, 1, out, lse, stream);
}

zsaa_status zsaa_op_attention_ex(const void* qkv, int B, int N, int Hq, int Hkv, int hd, int dtype,
                                 int causal, void* out, float* lse, zsaa_stream stream) {
  if (qkv == nullptr || out == nullptr || lse == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv) return fail(ZSAA_ERR_INVALID_ARG, "bad shape");
  if (dtype == ZSAA_BF16 && hd != 64 && hd != 128) return fail(ZSAA_ERR_UNSUPPORTED, "bf16 attention needs hd 64 or 128");
  if (dtype == ZSAA_F32 && (hd < 1 || hd > 128)) return fail(ZSAA_ERR_UNSUPPORTED, "f32 attention needs hd <= 128");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* status = shared_status();
  if (attention_pp_supported(dtype, hd, Hq, Hkv, nullptr, nullptr, status)) {
    ZCK(launch_attention_pp(qkv, B, N, Hq, Hkv, hd, out, lse, causal ? 1 : 0, status, s));
    return ZSAA_OK;
  }
  if (dtype == ZSAA_BF16 && status != nullptr) {  // the one-tile tcgen05 kernel, V^T scratch
    void* vt = nullptr;
    ZCK(cudaMallocAsync(&vt, attention_tc_vt_elems(B, N, Hkv, hd) * 2, s));
    cudaError_t e = launch_attention_tc(qkv, vt, B, N, Hq, Hkv, hd, out, lse, causal ? 1 : 0, status, s);
    cudaError_t e2 = cudaFreeAsync(vt, s);
    ZCK(e);
    ZCK(e2);
    return ZSAA_OK;
  }
  ZCK(launch_attention(dtype, qkv, B, N, Hq, Hkv, hd, out, lse, causal ? 1 : 0, s));
  return ZSAA_OK;
}

zsaa_status zsaa_op_colmass(const void* qkv, const float* lse, int B, int N, int Hq, int Hkv,
                            int hd, int dtype, float* colmass, zsaa_stream stream) {
  return zsaa_op_colmass_ex(qkv, lse, B, N, Hq, Hkv, hd, dtype, 1, colmass, stream);
}

zsaa_status zsaa_op_colmass_ex(const void* qkv, const float* lse, int B, int N, int Hq, int Hkv,
                               int hd, int dtype, int causal, float* colmass, zsaa_stream stream) {
  if (qkv == nullptr || lse == nullptr || colmass == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null argument");
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv) return fail(ZSAA_ERR_INVALID_ARG, "bad shape");
  if (dtype == ZSAA_BF16 && hd != 64 && hd != 128) return fail(ZSAA_ERR_UNSUPPORTED, "bf16 column mass needs hd 64 or 128");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  float* parts = nullptr;
  int* status = shared_status();
  if (status == nullptr) return fail(ZSAA_ERR_CUDA, "status word allocation failed");
  ZCK(cudaMallocAsync(reinterpret_cast<void**>(&parts),
                      colmass_parts_elems(B, N, Hq, Hkv) * sizeof(float), s));
  cudaError_t e = launch_colmass(dtype, qkv, lse, B, N, Hq, Hkv, hd, parts, colmass, status,
                                 causal ? 1 : 0, s);
  cudaError_t e2 = cudaFreeAsync(parts, s);
  ZCK(e);
  ZCK(e2);
  return ZSAA_OK;
}

zsaa_status zsaa_trace_begin(zsaa_model* m) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  m->trace.clear();
  m->ev_used = 0;
  m->trace_names.clear();
  m->tracing = true;
  return ZSAA_OK;
}

zsaa_status zsaa_trace_end(zsaa_model* m, zsaa_trace_row* rows, int max_rows, int* n_rows) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  m->tracing = false;
  ZCK(cudaDeviceSynchronize());
  std::vector<zsaa_trace_row> agg(m->trace_names.size());
  for (size_t i = 0; i < agg.size(); ++i) {
    memset(&agg[i], 0, sizeof(zsaa_trace_row));
    snprintf(agg[i].name, sizeof(agg[i].name), "%s", m->trace_names[i].c_str());
  }
  for (const auto& r : m->trace) {
    float ms = 0.f;
    ZCK(cudaEventElapsedTime(&ms, r.a, r.b));
    zsaa_trace_row& a = agg[r.cls];
    a.launches += r.kernels;
    a.ms += ms;
    a.flops += r.flops;
    a.bytes += r.bytes;
  }
  const int n = static_cast<int>(agg.size());
  if (n_rows) *n_rows = n;
  for (int i = 0; i < n && i < max_rows && rows != nullptr; ++i) rows[i] = agg[i];
  m->trace.clear();
  m->ev_used = 0;
  return ZSAA_OK;
}

zsaa_status zsaa_forward_masked(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                                float* logits_out, int32_t* kept_pos_out,
                                const zsaa_forward_opts* opts, zsaa_stream stream) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  return run_forward_masked(m, token_ids, B, L, accel, logits_out, kept_pos_out, opts,
                            reinterpret_cast<cudaStream_t>(stream));
}

zsaa_status zsaa_forward_marked(zsaa_model* m, const int32_t* token_ids, int B, int L, double accel,
                                float* logits_out, int32_t* kept_pos_out,
                                const zsaa_forward_opts* opts, zsaa_stream stream) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  return run_forward_masked(m, token_ids, B, L, accel, logits_out, kept_pos_out, opts,
                            reinterpret_cast<cudaStream_t>(stream), true);
}

zsaa_status zsaa_plan_varlen_config(const zsaa_config* cfg, const int32_t* lengths, int B,
                                    double accel, int* sched_out, double* alpha_out) {
  if (cfg == nullptr || sched_out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null config or output");
  zsaa_status st = validate_config(*cfg);
  if (st != ZSAA_OK) return st;
  return plan_varlen_impl(*cfg, lengths, B, accel, sched_out, alpha_out);
}

zsaa_status zsaa_plan_varlen(const zsaa_model* m, const int32_t* lengths, int B, double accel,
                             int* sched_out, double* alpha_out) {
  if (m == nullptr || sched_out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model or output");
  return plan_varlen_impl(m->cfg, lengths, B, accel, sched_out, alpha_out);
}

zsaa_status zsaa_forward_varlen(zsaa_model* m, const int32_t* token_ids, const int32_t* lengths,
                                int B, double accel, float* logits_out, int32_t* kept_pos_out,
                                const zsaa_forward_opts* opts, zsaa_stream stream) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  return run_forward_varlen(m, token_ids, lengths, B, accel, logits_out, kept_pos_out, opts,
                            reinterpret_cast<cudaStream_t>(stream));
}

zsaa_status zsaa_cache_create(zsaa_model* m, int B, int L, double accel, int max_new,
                              zsaa_cache** out) {
  if (out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null out");
  *out = nullptr;
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  const zsaa_config& c = m->cfg;
  if (c.dtype != ZSAA_BF16 || c.n_classes != 0 || !c.force_keep_last || c.bidirectional)
    return fail(ZSAA_ERR_UNSUPPORTED,
                "generation needs a causal bf16 model with the LM head and force_keep_last");
  if (B < 1 || B > m->max_B || L < 1 || L > m->max_L)
    return fail(ZSAA_ERR_INVALID_ARG, "B=%d L=%d outside [1,%d] x [1,%d]", B, L, m->max_B, m->max_L);
  if (max_new < 1 || max_new > (1 << 20))
    return fail(ZSAA_ERR_INVALID_ARG, "max_new=%d outside [1, 2^20]", max_new);
  if (c.n_heads % c.n_kv_heads != 0 || (c.n_heads / c.n_kv_heads) > 8 ||
      ((c.n_heads / c.n_kv_heads) & (c.n_heads / c.n_kv_heads - 1)) != 0 ||
      (c.head_dim != 64 && c.head_dim != 128))
    return fail(ZSAA_ERR_UNSUPPORTED, "generation supports head_dim 64/128 and 1/2/4/8 query heads per KV head");
  std::vector<int> sched(c.n_layers + 1);
  double alpha = 1.0;
  zsaa_status st = plan_impl(c, L, accel, sched.data(), &alpha);
  if (st != ZSAA_OK) return st;
  zsaa_cache* kc = new zsaa_cache();
  kc->m = m;
  kc->B = B;
  kc->L = L;
  kc->max_new = max_new;
  kc->accel = accel;
  kc->alpha = alpha;
  kc->sched = sched;
  const int Hkv = c.n_kv_heads, hd = c.head_dim;
  size_t kv_elems = 0, pos_elems = 0;
  for (int l = 1; l <= c.n_layers; ++l) {
    const size_t cap = static_cast<size_t>(sched[l - 1]) + max_new;
    kv_elems += 2 * static_cast<size_t>(B) * Hkv * cap * hd;
    pos_elems += static_cast<size_t>(B) * cap;
  }
  kc->kv_bytes = kv_elems * 2;
  kc->kv_bytes_unpruned = static_cast<size_t>(c.n_layers) * 2 * B * Hkv * (static_cast<size_t>(L) + max_new) * hd * 2;
  bool ok = true;
  auto alloc = [&](void** p, size_t bytes) {
    if (ok && cudaMalloc(p, bytes + 16) != cudaSuccess) ok = false;
  };
  const int n_pos = L + max_new;
  alloc(&kc->kv, kv_elems * 2);
  alloc(reinterpret_cast<void**>(&kc->pos), pos_elems * sizeof(int32_t));
  alloc(reinterpret_cast<void**>(&kc->rope_cos), static_cast<size_t>(n_pos) * (hd / 2) * sizeof(float));
  alloc(reinterpret_cast<void**>(&kc->rope_sin), static_cast<size_t>(n_pos) * (hd / 2) * sizeof(float));
  alloc(reinterpret_cast<void**>(&kc->qkv32), static_cast<size_t>(B) * m->ld_qkv * sizeof(float));
  alloc(reinterpret_cast<void**>(&kc->last_idx), static_cast<size_t>(B) * sizeof(int32_t));
  alloc(reinterpret_cast<void**>(&kc->step), sizeof(int));
  if (!ok) {
    cudaGetLastError();
    const size_t want = kc->kv_bytes;
    free_cache(kc);
    return fail(ZSAA_ERR_OOM, "cache allocation failed (%zu bytes of keys/values)", want);
  }
  size_t off_kv = 0, off_pos = 0;
  for (int l = 1; l <= c.n_layers; ++l) {
    const int cap = sched[l - 1] + max_new;
    const size_t plane = static_cast<size_t>(B) * Hkv * cap * hd;
    zsaa::KvLayer kl;
    kl.k = static_cast<uint16_t*>(kc->kv) + off_kv;
    kl.v = static_cast<uint16_t*>(kc->kv) + off_kv + plane;
    kl.pos = kc->pos + off_pos;
    kl.cap = cap;
    kl.base = sched[l - 1];
    kc->layers.push_back(kl);
    off_kv += 2 * plane;
    off_pos += static_cast<size_t>(B) * cap;
  }
  std::vector<float> cs, sn;
  rope_host_table(c.rope_theta, hd, n_pos, &cs, &sn);
  std::vector<int32_t> last(B, sched[c.n_layers] - 1);
  cudaError_t e = cudaMemcpy(kc->rope_cos, cs.data(), cs.size() * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(kc->rope_sin, sn.data(), sn.size() * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(kc->last_idx, last.data(), last.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(kc->step, 0, sizeof(int));
  if (e != cudaSuccess) {
    free_cache(kc);
    return fail(ZSAA_ERR_CUDA, "cache initialisation failed: %s", cudaGetErrorString(e));
  }
  *out = kc;
  return ZSAA_OK;
}

void zsaa_cache_destroy(zsaa_cache* c) {
  if (c == nullptr) return;
  cudaDeviceSynchronize();
  zsaa_model* m = c->m;
  for (auto it = m->graphs.begin(); it != m->graphs.end();) {  // graphs that use this cache
    if (it->cache == c) {
      if (it->exec) cudaGraphExecDestroy(it->exec);
      it = m->graphs.erase(it);
    } else {
      ++it;
    }
  }
  free_cache(c);
}

zsaa_status zsaa_prefill(zsaa_model* m, zsaa_cache* c, const int32_t* token_ids,
                         float* logits_out, const zsaa_forward_opts* opts, zsaa_stream stream) {
  if (m == nullptr || c == nullptr || c->m != m) return fail(ZSAA_ERR_INVALID_ARG, "null model/cache or cache of another model");
  if (token_ids == nullptr || logits_out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null token or logits pointer");
  if (opts && (opts->hidden_out || opts->n_layers_run || opts->hidden_in || opts->pos_in ||
               opts->first_layer || opts->plan_L))
    return fail(ZSAA_ERR_INVALID_ARG, "zsaa_prefill takes only the forced_idx/scores_out/idx_out hooks");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  ZCK(cudaMemsetAsync(c->step, 0, sizeof(int), s));
  zsaa_status st;
  if (opts && (opts->forced_idx || opts->scores_out || opts->idx_out))
    st = run_forward(m, token_ids, c->B, c->L, c->accel, logits_out, nullptr, opts, s, c);
  else
    st = forward_cached(m, token_ids, c->B, c->L, c->accel, logits_out, nullptr, s, c);
  if (st == ZSAA_OK) {
    c->generated = 0;
    c->prefilled = true;
  }
  return st;
}

zsaa_status zsaa_decode_step(zsaa_model* m, zsaa_cache* c, const int32_t* token_ids,
                             float* logits_out, zsaa_stream stream) {
  if (m == nullptr || c == nullptr || c->m != m) return fail(ZSAA_ERR_INVALID_ARG, "null model/cache or cache of another model");
  if (token_ids == nullptr || logits_out == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null token or logits pointer");
  if (!c->prefilled) return fail(ZSAA_ERR_INVALID_ARG, "zsaa_decode_step before zsaa_prefill");
  if (c->generated >= c->max_new)
    return fail(ZSAA_ERR_INVALID_ARG, "cache full: %d tokens generated, max_new %d", c->generated, c->max_new);
  zsaa_status st = decode_cached(m, c, token_ids, logits_out, reinterpret_cast<cudaStream_t>(stream));
  if (st == ZSAA_OK) c->generated += 1;
  return st;
}

zsaa_status zsaa_cache_layer(const zsaa_cache* c, int layer, void** k, void** v, int32_t** pos,
                             int* base, int* len, int* cap) {
  if (c == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null cache");
  if (layer < 1 || layer > static_cast<int>(c->layers.size()))
    return fail(ZSAA_ERR_INVALID_ARG, "layer %d outside [1, %zu]", layer, c->layers.size());
  const zsaa::KvLayer& l = c->layers[layer - 1];
  if (k) *k = l.k;
  if (v) *v = l.v;
  if (pos) *pos = l.pos;
  if (base) *base = l.base;
  if (len) *len = l.base + c->generated;
  if (cap) *cap = l.cap;
  return ZSAA_OK;
}

zsaa_status zsaa_cache_bytes(const zsaa_cache* c, size_t* pruned, size_t* unpruned) {
  if (c == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null cache");
  if (pruned) *pruned = c->kv_bytes;
  if (unpruned) *unpruned = c->kv_bytes_unpruned;
  return ZSAA_OK;
}

zsaa_status zsaa_sync(zsaa_model* m, zsaa_stream stream) {
  if (m == nullptr) return fail(ZSAA_ERR_INVALID_ARG, "null model");
  return read_status(m->status, reinterpret_cast<cudaStream_t>(stream), false);
}

zsaa_status zsaa_device_status(void) {
  int* w = shared_status();
  if (w == nullptr) return fail(ZSAA_ERR_CUDA, "status word allocation failed");
  return read_status(w, nullptr, true);
}

zsaa_status zsaa_selftest_wait_timeout(zsaa_stream stream) {
  int* w = shared_status();
  if (w == nullptr) return fail(ZSAA_ERR_CUDA, "status word allocation failed");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  wait_timeout_selftest_kernel<<<1, 64, 0, s>>>(w);
  ZCK(cudaGetLastError());
  return read_status(w, s, false);
}

}  // extern "C"
