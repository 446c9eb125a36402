// SD^2 engine: host orchestration of one draft-and-verify iteration behind the C ABI of sd2.h.
//
//   sd2_prefill  verifier over the prompts -> first token (bonus-style sample at step 0) ->
//                steering from the last prompt row -> drafter over the prompts under its biases
//   sd2_step     a1 steering (Sec. 3.1, App. A.2) -> a2 k drafter steps with Eq. 2 biases ->
//                a3 verifier over the k+1 block rows, writing taps and logits
//   sd2_accept   a4 acceptance (Sec. 3.1) -> commit and rollback of both caches
//
// All per-sequence lengths live on the device (state.cu), so step and accept are each captured
// once into a CUDA graph and replayed. The decoder forward is a fixed chain per layer:
// RMSNorm(+taps) -> QKV GEMM -> rotary + paged KV append -> attention -> O GEMM (+residual) ->
// RMSNorm -> gate/up GEMM with the steered SwiGLU epilogue -> down GEMM (+residual).
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <string>
#include <vector>

#include "sd2.h"
#include "common.cuh"
#include "kernels.h"
#include "state.h"
#include "tc.cuh"

using namespace sd2;

namespace {

thread_local std::string g_last_error;

struct Model {
  sd2_lm_config c{};
  const void* embed = nullptr;
  const void* final_norm = nullptr;
  const void* lm_head = nullptr;
  std::vector<const void*> w;
  void* kv_pool = nullptr;
  int* table = nullptr;
  int bt_stride = 0, n_blocks = 0;
  float* rope_cs = nullptr;
  const void* W(int l, int s) const { return w[static_cast<size_t>(l) * SD2_LAYER_SLOTS + s]; }
  int qkv_width() const { return (c.n_heads + 2 * c.n_kv_heads) * c.head_dim; }
  int group_rows() const { return std::max(1, 64 / (c.n_heads / c.n_kv_heads)); }
  KVCache cache() const {
    KVCache k;
    k.pool = kv_pool; k.table = table; k.bt_stride = bt_stride; k.n_blocks = n_blocks;
    k.Hkv = c.n_kv_heads; k.hd = c.head_dim;
    return k;
  }
};

struct Plan {
  int M = 0;
  const int* tok = nullptr;
  const int* pos = nullptr;
  const int* seq = nullptr;
  const int* valid = nullptr;
  int n_groups = 0;
  const int* g_row0 = nullptr;
  const int* g_nrows = nullptr;
  const int* g_seq = nullptr;
  int n_splits = 1, chunk = 64;
  int max_rows = 1;  // rows of the largest attention group
  // decode steps: the pre-step lengths attention may read before its programmatic wait (AttnArgs)
  const int* pre_len = nullptr;
  int pre_stable = 0, pre_fresh = 0;
};

struct ProfRec {
  int cls;
  double bytes;
  cudaEvent_t e0, e1;
};

}  // namespace

struct sd2_ctx {
  sd2_config cfg{};
  Model V, D;
  const void *w_hml = nullptr, *ln_g = nullptr, *ln_b = nullptr, *w_s = nullptr;
  const void *w_c1x = nullptr, *w_c1g = nullptr, *w_c2 = nullptr;   // steering_site 2
  cudaStream_t st = nullptr, cap_st = nullptr;
  int B = 0, phase = 0, maxB = 0, max_rows = 0;
  unsigned long long seed = 0;
  unsigned long long* seed_d = nullptr;   // the request's seed on the device, read by the captured step
  std::vector<int> graph_key;             // batch, k and the step-shape tables the captured graphs were built on
  std::string err;
  std::vector<void*> allocs;
  // device state
  int *state = nullptr, *committed = nullptr, *iter = nullptr, *xhat = nullptr;
  float* temp = nullptr;
  unsigned* errw = nullptr;
  int *row_tok = nullptr, *row_pos = nullptr, *row_seq = nullptr, *row_valid = nullptr;
  int* statics = nullptr;  // group tables and row lists of the step shapes, then prefill's
  int statics_cap = 0;
  // activations
  float *x = nullptr, *qkv = nullptr, *q = nullptr, *logits_t = nullptr, *logits_d = nullptr;
  float *taps = nullptr, *g_pre = nullptr, *g = nullptr, *bias = nullptr;
  float* ssq = nullptr;          // fused RMSNorm: [slices][max_rows] sums of squares of the residual stream
  // steering_site 2: per-stage W_c1g g [B, L_D*d_g], per-layer f^(l-1) in bf16 [R, d_D], the bias
  // MLP's hidden layer [R, d_g] and its per-row output [R, F_D]; row index table [R]
  float* cg = nullptr;
  void* fb = nullptr;
  void* cu_h = nullptr;
  float* rowbias = nullptr;
  int* row_ident = nullptr;
  ChainPlan chain{};             // the drafter's persistent layer chain (chain.cu), when its shape allows
  bool chain_ok = false;
  bool use_chain = false;        // measured slower than the per-kernel path on GB300 (off by default)
  bool attn_in_o = false;        // decode attention inside the O projection: measured slower on GB300 (off by default)
  void *a = nullptr, *attn = nullptr, *h = nullptr, *g_bf = nullptr, *hml_in = nullptr;
  // long-context attention: partials of the context clusters and the per-share arrival counters
  void *attn_part_acc = nullptr, *attn_part_ml = nullptr, *attn_part_cnt = nullptr;
  void *attn_flat_acc = nullptr, *attn_flat_ml = nullptr;   // flat-mode attention partials
  unsigned* attn_flat_cnt = nullptr;
  int gemm_impl = 0;            // 0 tensor cores where the shape allows, 1 CUDA cores
  unsigned long long* samp_slot = nullptr;
  int* samp_counter = nullptr;
  AcceptScratch as{};
  int *tok_out = nullptr, *n_out = nullptr, *first = nullptr, *cu = nullptr;
  // sd2_generate: the prompt on the device, the emitted tokens of a step, and their pinned host copy
  int *gen_prompt = nullptr, *gen_first = nullptr, *gen_tok = nullptr, *gen_n = nullptr;
  int* gen_host = nullptr;
  // step-shape plans
  Plan p_d1, p_dn, p_v;
  const int* logit_rows_d1 = nullptr;
  // graphs
  bool use_graphs = true;
  cudaGraphExec_t g_step = nullptr, g_accept = nullptr;
  // profiling
  bool prof = false;
  bool stage_on = false;                  // stage markers inside the step (graph event nodes)
  bool stage_done = false;
  std::vector<cudaEvent_t> stage_ev;      // [k + 3]: before steer, after steer, after draft i, after verify
  // in-graph GEMM timing: globaltimer stamps of every tensor-core GEMM launch of the step
  bool gemm_timing = false;
  bool gemm_timing_done = false;
  unsigned long long* gstamp = nullptr;   // [kMaxStampedLaunches][3] (GemmArgs::stamp)
  int gstamp_n = 0;                       // launches stamped by the step being enqueued
  int cur_stage = -1;                     // 0 steering, 1..k drafter step i, k + 1 verify
  std::vector<double> gstamp_bytes;
  std::vector<int> gstamp_stage;
  std::vector<ProfRec> recs;
  std::vector<cudaEvent_t> ev_pool;
  std::vector<int> h_n;  // host copy of committed lengths while profiling
};

// ------------------------------------------------------------------------------------------------
// helpers
// ------------------------------------------------------------------------------------------------
namespace {

sd2_status fail(sd2_ctx* c, sd2_status s, const std::string& m) {
  if (c) c->err = m;
  g_last_error = m;
  return s;
}

#define CK(call)                                                                                   \
  do {                                                                                             \
    cudaError_t e_ = (call);                                                                       \
    if (e_ != cudaSuccess) return fail(c, SD2_ECUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

// Test hook (sd2_debug_fail_alloc): the number of context allocations still to succeed before
// one is made to fail; -1 when disarmed.
std::atomic<int> g_fail_alloc_after{-1};

bool injected_alloc_failure() {
  int cur = g_fail_alloc_after.load();
  while (cur >= 0 && !g_fail_alloc_after.compare_exchange_weak(cur, cur - 1)) {
  }
  return cur == 0;
}

template <typename T>
sd2_status dalloc(sd2_ctx* c, T** p, size_t n) {
  void* v = nullptr;
  const size_t bytes = std::max<size_t>(n * sizeof(T), 256);
  if (injected_alloc_failure())
    return fail(c, SD2_ENOMEM, "cudaMalloc of " + std::to_string(bytes) + " bytes failed (injected by sd2_debug_fail_alloc)");
  if (cudaMalloc(&v, bytes) != cudaSuccess) {
    cudaGetLastError();
    return fail(c, SD2_ENOMEM, "cudaMalloc of " + std::to_string(bytes) + " bytes failed");
  }
  c->allocs.push_back(v);
  *p = static_cast<T*>(v);
  return SD2_OK;
}
#define ALLOC(p, n)                                  \
  do {                                               \
    sd2_status s_ = dalloc(c, &(p), (size_t)(n));    \
    if (s_ != SD2_OK) return s_;                     \
  } while (0)

cudaEvent_t take_event(sd2_ctx* c) {
  cudaEvent_t e;
  if (!c->ev_pool.empty()) {
    e = c->ev_pool.back();
    c->ev_pool.pop_back();
  } else {
    cudaEventCreate(&e);
  }
  return e;
}

// Run `fn` (which enqueues on c->st) and, when profiling, bracket it with events.
template <typename F>
cudaError_t timed(sd2_ctx* c, int cls, double bytes, F fn) {
  if (!c->prof) return fn();
  ProfRec r{cls, bytes, take_event(c), take_event(c)};
  cudaEventRecord(r.e0, c->st);
  cudaError_t e = fn();
  cudaEventRecord(r.e1, c->st);
  c->recs.push_back(r);
  return e;
}
constexpr int kMaxCtxClusters = 4;   // context clusters of one long-context attention launch
constexpr int kMaxFlatGroups = 64;   // row groups of one flat-mode attention launch
// Fewest row groups, and rows per group, for flat mode. Balancing pays where the tile loop
// dominates: the batch-16 verify (9 rows a group, 128-1280 positions) went from 5.95 to 5.73 ms,
// while its drafter steps (1-2 rows a group) went from 0.939 to 0.961 ms and 4 sequences of equal
// length (the Qwen pair) gained nothing, the merge through global memory costing more than the
// cluster's.
constexpr int kMinFlatGroups = 8;
constexpr int kMinFlatRows = 4;
constexpr int kMaxCtxGroups = 4;     // attention row groups a launch with context clusters may have
constexpr int kMaxStampedLaunches = 8192;   // GEMM launches of one step that in-graph timing can follow
enum { PC_GEMM = 0, PC_ATTN = 1, PC_ACCEPT = 2, PC_SAMPLE = 3, PC_OTHER = 4, PC_VERIFY = 5, PC_DRAFT = 6, PC_STEER = 7,
       PC_N = 8 };

bool valid_lm(const sd2_lm_config& m) {
  return m.n_layers > 0 && m.d_model > 0 && m.d_model % 8 == 0 && (m.head_dim == 64 || m.head_dim == 128) &&
         m.n_heads > 0 && m.n_kv_heads > 0 && m.n_heads % m.n_kv_heads == 0 && m.n_heads / m.n_kv_heads <= 64 &&
         m.d_ffn > 0 && m.d_ffn % 8 == 0 && m.vocab > 0 && m.vocab % 4 == 0 && m.rope_theta > 0 && m.norm_eps > 0;
}
bool aligned16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

sd2_status load_model(sd2_ctx* c, Model& m, const sd2_lm_config& cfg, const sd2_lm_weights& w, const char* name) {
  m.c = cfg;
  if (!aligned16(w.embed) || !aligned16(w.final_norm) || !aligned16(w.lm_head) || !w.layers)
    return fail(c, SD2_EINVAL, std::string(name) + ": null or unaligned embed/final_norm/lm_head/layers");
  m.embed = w.embed; m.final_norm = w.final_norm; m.lm_head = w.lm_head;
  m.w.assign(w.layers, w.layers + static_cast<size_t>(cfg.n_layers) * SD2_LAYER_SLOTS);
  for (size_t i = 0; i < m.w.size(); ++i)
    if (!aligned16(m.w[i]))
      return fail(c, SD2_EINVAL, std::string(name) + ": layer weight " + std::to_string(i) + " null or not 16-byte aligned");
  const int maxB = c->cfg.max_batch;
  m.bt_stride = (c->cfg.max_ctx + 15) / 16;
  m.n_blocks = maxB * m.bt_stride;
  const size_t kv_elems = static_cast<size_t>(cfg.n_layers) * m.n_blocks * 2 * cfg.n_kv_heads * 16 * cfg.head_dim;
  void* pool;
  ALLOC(pool, kv_elems * 2);
  m.kv_pool = pool;
  int* table;
  ALLOC(table, static_cast<size_t>(maxB) * m.bt_stride);
  m.table = table;
  std::vector<int> ht(static_cast<size_t>(maxB) * m.bt_stride);
  for (int b = 0; b < maxB; ++b)       // block i of sequence b: interleaved across sequences
    for (int i = 0; i < m.bt_stride; ++i) ht[static_cast<size_t>(b) * m.bt_stride + i] = i * maxB + b;
  CK(cudaMemcpy(table, ht.data(), ht.size() * sizeof(int), cudaMemcpyHostToDevice));
  CK(cudaMemset(pool, 0, kv_elems * 2));
  const int half = cfg.head_dim / 2;
  std::vector<float> cs(static_cast<size_t>(c->cfg.max_ctx) * half * 2);
  for (int p = 0; p < c->cfg.max_ctx; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = p * pow(static_cast<double>(cfg.rope_theta), -2.0 * i / cfg.head_dim);
      cs[(static_cast<size_t>(p) * half + i) * 2] = static_cast<float>(cos(ang));
      cs[(static_cast<size_t>(p) * half + i) * 2 + 1] = static_cast<float>(sin(ang));
    }
  float* rcs;
  ALLOC(rcs, cs.size());
  m.rope_cs = rcs;
  CK(cudaMemcpy(rcs, cs.data(), cs.size() * sizeof(float), cudaMemcpyHostToDevice));
  return SD2_OK;
}

// ------------------------------------------------------------------------------------------------
// forward of one decoder over a row plan
// ------------------------------------------------------------------------------------------------
struct FwdOut {
  const float* bias = nullptr;    // [*, L*F] steering biases (drafter) or null
  float* taps = nullptr;          // [rows, 3, d] (verifier) or null
  const int* tap_row = nullptr;
  int tap_layers[3] = {0, 0, 0};
  const int* logit_rows = nullptr;
  int n_logit_rows = 0;
  float* logits = nullptr;
  long long ld_logits = 0;
};

// The error word and the implementation choice, attached to every GEMM launch.
GemmArgs& tc(sd2_ctx* c, GemmArgs& g) {
  g.err = c->errw;
  g.impl = c->gemm_impl;
  return g;
}

// One GEMM launch of the hot path: bracketed by events when profiling, and given a globaltimer
// stamp slot when in-graph GEMM timing is on (bytes = its algorithmic bytes).
sd2_status run_gemm(sd2_ctx* c, GemmArgs& g, double bytes) {
  tc(c, g);
  if (c->gemm_timing && c->gstamp && c->gstamp_n < kMaxStampedLaunches) {
    g.stamp = c->gstamp + 3 * static_cast<size_t>(c->gstamp_n++);
    c->gstamp_bytes.push_back(bytes);
    c->gstamp_stage.push_back(c->cur_stage);
  }
  CK(timed(c, PC_GEMM, bytes, [&] { return gemm(g, c->st); }));
  return SD2_OK;
}
#define RUN_GEMM(g, bytes)                        \
  do {                                            \
    sd2_status s_ = run_gemm(c, (g), (bytes));    \
    if (s_ != SD2_OK) return s_;                  \
  } while (0)

// Steering bias entries per drafter layer: F_D for Eq. 2 (inside the MLP), d_D after the MLP.
int bias_width(const sd2_ctx* c) { return c->cfg.steering_site ? c->D.c.d_model : c->D.c.d_ffn; }

double gemm_bytes(int M, int N, int K, int out_bytes) {
  return 2.0 * N * K + 2.0 * M * K + static_cast<double>(out_bytes) * M * N;
}

// Final RMSNorm (with the last tap) and lm_head over the logit rows, from the residual stream c->x.
// Final RMSNorm and lm_head. final_parts > 0: the last layer's down projection already produced
// bf16(x * gamma_final), the last taps and final_parts slices of the sums of squares (every row
// takes logits), so the lm_head applies the norm's row scale itself.
sd2_status head(sd2_ctx* c, const Model& m, const Plan& p, const FwdOut& o, int final_parts = 0) {
  const sd2_lm_config& mc = m.c;
  const int M = p.M, d = mc.d_model, L = mc.n_layers;
  int mask = 0;
  if (o.taps)
    for (int s = 0; s < 3; ++s)
      if (o.tap_layers[s] == L) mask |= 1 << s;
  if (final_parts == 0 && (o.n_logit_rows > 0 || mask)) {
    const int nr = o.n_logit_rows > 0 ? o.n_logit_rows : M;
    CK(timed(c, PC_OTHER, 0, [&] {
      return rmsnorm(c->x, o.logit_rows, m.final_norm, mc.norm_eps, nr, d, c->a, o.taps, o.tap_row, mask, c->st);
    }));
  }
  if (o.n_logit_rows > 0) {
    GemmArgs gl{};
    gl.x = c->a; gl.ldx = d; gl.M = o.n_logit_rows; gl.K = d;
    gl.seg[0] = {m.lm_head, mc.vocab}; gl.nseg = 1; gl.epi = EPI_STORE; gl.out = o.logits;
    gl.ldo = static_cast<int>(o.ld_logits);
    if (final_parts > 0) {
      gl.norm_ssq_in = c->ssq; gl.norm_parts = final_parts; gl.norm_d = d; gl.norm_eps = mc.norm_eps;
      gl.ld_ssq = c->max_rows;
    }
    RUN_GEMM(gl, gemm_bytes(o.n_logit_rows, mc.vocab, d, 4));
  }
  return SD2_OK;
}

// The drafter's layers over plan p in one persistent launch (chain.cu), then the head. Used for
// the drafter steps when the chain takes their shape; forward() otherwise.
bool chain_takes(sd2_ctx* c, const Plan& p) {
  if (!c->chain_ok || !c->use_chain || c->gemm_impl != 0 || c->cfg.steering_site != 0) return false;
  ChainRun r;
  r.M = p.M; r.n_splits = p.n_splits; r.chunk = p.chunk; r.max_rows = p.max_rows;
  return chain_supported(c->chain, r);
}
sd2_status forward_chain(sd2_ctx* c, const Model& m, const Plan& p, const FwdOut& o) {
  ChainRun r;
  r.M = p.M; r.tok = p.tok; r.row_pos = p.pos; r.row_seq = p.seq; r.row_valid = p.valid;
  r.grp_row0 = p.g_row0; r.grp_nrows = p.g_nrows; r.grp_seq = p.g_seq; r.n_groups = p.n_groups;
  r.n_splits = p.n_splits; r.chunk = p.chunk; r.max_rows = p.max_rows;
  r.bias = o.bias; r.ld_bias = m.c.n_layers * m.c.d_ffn;
  r.x_out = c->x; r.err = c->errw;
  double bytes = 0;
  if (c->prof) {
    const sd2_lm_config& mc = m.c;
    bytes = 2.0 * mc.n_layers * (static_cast<double>(mc.d_model) * m.qkv_width() +
                                 static_cast<double>(mc.n_heads) * mc.head_dim * mc.d_model + 3.0 * mc.d_model * mc.d_ffn);
  }
  CK(timed(c, PC_GEMM, bytes, [&] { return chain_forward(c->chain, r, c->st); }));
  return head(c, m, p, o);
}

// Decoder forward pass over the rows of plan p. On the tensor-core path the RMSNorm in front of
// each projection is fused into the GEMMs around it: the residual-adding GEMM (or the embedding)
// that produces x also writes bf16(x * gamma) and per-slice sums of squares of x, and the next
// GEMM scales its outputs by the row's rsqrt(mean(x^2) + eps). Otherwise separate RMSNorm
// kernels run between the GEMMs.
sd2_status forward(sd2_ctx* c, const Model& m, const Plan& p, const FwdOut& o) {
  const sd2_lm_config& mc = m.c;
  const int M = p.M, d = mc.d_model, H = mc.n_heads, Hkv = mc.n_kv_heads, hd = mc.head_dim, F = mc.d_ffn;
  const int L = mc.n_layers;
  const int R = c->max_rows;
  auto tap_mask = [&](int layer_out) {
    int mask = 0;
    if (!o.taps) return 0;
    for (int s = 0; s < 3; ++s)
      if (o.tap_layers[s] == layer_out) mask |= 1 << s;
    return mask;
  };
  auto qkv_args = [&](int l) {
    GemmArgs g{};
    g.x = c->a; g.ldx = d; g.M = M; g.K = d;
    g.seg[0] = {m.W(l, SD2_W_Q), H * hd};
    g.seg[1] = {m.W(l, SD2_W_K), Hkv * hd};
    g.seg[2] = {m.W(l, SD2_W_V), Hkv * hd};
    g.nseg = 3; g.epi = EPI_QKV; g.out = c->qkv; g.ldo = m.qkv_width();
    g.q_out = c->q; g.kv_pool = m.kv_pool; g.kv_table = m.table; g.kv_bt_stride = m.bt_stride;
    g.kv_n_blocks = m.n_blocks; g.n_heads = H; g.n_kv_heads = Hkv; g.head_dim = hd; g.layer = l;
    g.rope_cs = m.rope_cs; g.row_pos = p.pos; g.row_valid = p.valid; g.row_seq = p.seq;
    return g;
  };
  auto o_args = [&](int l) {
    GemmArgs g{};
    g.x = c->attn; g.ldx = H * hd; g.M = M; g.K = H * hd;
    g.seg[0] = {m.W(l, SD2_W_O), d}; g.nseg = 1; g.epi = EPI_ADD; g.out = c->x; g.ldo = d;
    return g;
  };
  auto gu_args = [&](int l) {
    GemmArgs g{};
    g.x = c->a; g.ldx = d; g.M = M; g.K = d;
    g.seg[0] = {m.W(l, SD2_W_GATE), F}; g.seg[1] = {m.W(l, SD2_W_UP), F}; g.nseg = 2;
    g.epi = EPI_SWIGLU; g.out_bf = c->h; g.ldh = F;
    if (c->cfg.steering_site == 0) {     // Eq. 2: added to W_u a before the gating
      g.bias = o.bias ? o.bias + static_cast<size_t>(l) * F : nullptr;
      g.ld_bias = L * F;
    }
    g.row_seq = p.seq;
    return g;
  };
  auto down_args = [&](int l) {
    GemmArgs g{};
    g.x = c->h; g.ldx = F; g.M = M; g.K = F;
    g.seg[0] = {m.W(l, SD2_W_DOWN), d}; g.nseg = 1; g.epi = EPI_ADD; g.out = c->x; g.ldo = d;
    if (c->cfg.steering_site == 1 && o.bias) {   // after the MLP: added to the layer's output
      g.bias = o.bias + static_cast<size_t>(l) * d;
      g.ld_bias = L * d;
      g.row_seq = p.seq;
    }
    return g;
  };
  // producer / consumer halves of a fused RMSNorm with gamma
  auto produce = [&](GemmArgs& g, const void* gamma) {
    g.norm_gamma = gamma; g.norm_out = c->a; g.norm_ssq_out = c->ssq; g.ld_ssq = R;
  };
  auto consume = [&](GemmArgs& g, int parts) {
    g.norm_ssq_in = c->ssq; g.norm_parts = parts; g.norm_d = d; g.norm_eps = mc.norm_eps; g.ld_ssq = R;
  };
  bool fused = c->gemm_impl == 0 && tap_mask(0) == 0 && d % 128 == 0;
  if (fused) {
    GemmArgs g0 = qkv_args(0), g1 = o_args(0), g2 = gu_args(0), g3 = down_args(0);
    tc(c, g0); tc(c, g1); tc(c, g2); tc(c, g3);
    consume(g0, 1); produce(g1, m.W(0, SD2_W_MLP_NORM)); consume(g2, 1); produce(g3, m.W(0, SD2_W_ATTN_NORM));
    fused = gemm_tc_supported(g0) && gemm_tc_supported(g1) && gemm_tc_supported(g2) && gemm_tc_supported(g3) &&
            gemm_norm_parts(g1) <= (d / 128 + 1) * 8 && gemm_norm_parts(g3) <= (d / 128 + 1) * 8;
  }
  int parts = 1;   // slices of the sums of squares the last producer wrote
  // every row of the plan takes logits: the last down projection can produce the final norm too
  const bool final_in_down = o.n_logit_rows == M && o.logit_rows == nullptr && !o.tap_row;
  if (fused) {
    CK(timed(c, PC_OTHER, 0, [&] {
      return embed_scaled(p.tok, m.embed, m.W(0, SD2_W_ATTN_NORM), M, d, mc.vocab, c->x, c->a, c->ssq, c->st);
    }));
  } else {
    CK(timed(c, PC_OTHER, 0, [&] {
      return embed_rmsnorm(p.tok, m.embed, m.W(0, SD2_W_ATTN_NORM), mc.norm_eps, M, d, mc.vocab, c->x, c->a, c->st);
    }));
  }
  for (int l = 0; l < L; ++l) {
    if (l > 0 && !fused)
      CK(timed(c, PC_OTHER, 0, [&] {
        return rmsnorm(c->x, nullptr, m.W(l, SD2_W_ATTN_NORM), mc.norm_eps, M, d, c->a, o.taps, o.tap_row, tap_mask(l),
                       c->st);
      }));
    if (c->cfg.steering_site == 2 && o.bias) {
      // "Cond. Bias in MLP" (Sec. 5): b = W_c2 SiLU(W_c1x f^(l-1) + W_c1g g) per row, from this
      // layer's input f^(l-1) = x (before the attention) and the stage's W_c1g g
      const int dg = c->cfg.d_steer;
      CK(timed(c, PC_OTHER, 0, [&] { return rows_to_bf16(c->x, d, M, d, c->fb, c->st); }));
      GemmArgs c1{};
      c1.x = c->fb; c1.ldx = d; c1.M = M; c1.K = d;
      c1.seg[0] = {static_cast<const char*>(c->w_c1x) + static_cast<size_t>(l) * dg * d * 2, dg}; c1.nseg = 1;
      c1.epi = EPI_SILU; c1.out_bf = c->cu_h; c1.ldh = dg;
      c1.bias = c->cg + static_cast<size_t>(l) * dg; c1.ld_bias = L * dg; c1.row_seq = p.seq;
      RUN_GEMM(c1, gemm_bytes(M, dg, d, 2));
      GemmArgs c2{};
      c2.x = c->cu_h; c2.ldx = dg; c2.M = M; c2.K = dg;
      c2.seg[0] = {static_cast<const char*>(c->w_c2) + static_cast<size_t>(l) * F * dg * 2, F}; c2.nseg = 1;
      c2.epi = EPI_STORE; c2.out = c->rowbias; c2.ldo = F;
      RUN_GEMM(c2, gemm_bytes(M, F, dg, 4));
    }
    GemmArgs g = qkv_args(l);
    if (fused) consume(g, parts);
    RUN_GEMM(g, gemm_bytes(M, m.qkv_width(), d, 4));
    // A decode step of one sequence may run its attention inside the O projection (gemm_tc.cu).
    GemmArgs go = o_args(l);
    if (fused) produce(go, m.W(l, SD2_W_MLP_NORM));
    bool in_o = false;
    if (c->attn_in_o && p.pre_len && p.n_groups == 1 && c->gemm_impl == 0) {
      GemmArgs ga = go;
      ga.attn_q = c->q; ga.attn_seq = p.g_seq; ga.attn_pre_len = p.pre_len;
      ga.attn_pre_stable = p.pre_stable; ga.attn_pre_fresh = p.pre_fresh;
      ga.kv_pool = m.kv_pool; ga.kv_table = m.table; ga.kv_bt_stride = m.bt_stride; ga.kv_n_blocks = m.n_blocks;
      ga.n_heads = H; ga.n_kv_heads = Hkv; ga.head_dim = hd; ga.layer = l; ga.row_pos = p.pos;
      if (gemm_attn_supported(tc(c, ga))) {
        go = ga;
        in_o = true;
      }
    }
    if (fused) parts = gemm_norm_parts(go);
    AttnArgs at{};
    at.q = c->q; at.kv = m.cache(); at.layer = l; at.row_pos = p.pos;
    at.grp_row0 = p.g_row0; at.grp_nrows = p.g_nrows; at.grp_seq = p.g_seq; at.n_groups = p.n_groups;
    at.M = M; at.H = H; at.hd = hd; at.n_splits = p.n_splits; at.chunk = p.chunk; at.max_rows = p.max_rows; at.out = c->attn;
    if (p.pre_len) {   // decode step: as many context splits as the GPU holds resident at once, no more
      const long resident = static_cast<long>(attention_ctas_per_sm(hd)) * sm_count_cached();
      const int want = std::max(1, static_cast<int>(resident / std::max(1, p.n_groups * Hkv)));
      const int max_ctx = c->cfg.max_ctx;
      auto chunk_for = [max_ctx](int ns, int R) { return 64 * ((max_ctx + 64 * ns * R - 1) / (64 * ns * R)); };
      at.pre_len = p.pre_len;
      const int W = static_cast<int>(resident / Hkv);
      if (p.n_groups >= kMinFlatGroups && p.n_groups <= kMaxFlatGroups && p.max_rows >= kMinFlatRows &&
          W >= p.n_groups && max_ctx > 64) {
        // many row groups (sequences of ragged lengths) of several rows each: flat mode, every
        // resident CTA a slot, the slots shared out on the device by the sequences' lengths
        at.n_splits = 1;
        at.flat = W;
        at.chunk = 64 * ((max_ctx + 63) / 64);
        at.flat_acc = c->attn_flat_acc; at.flat_ml = c->attn_flat_ml; at.flat_cnt = c->attn_flat_cnt;
      } else if (want < at.n_splits) {
        at.n_splits = want;
        at.chunk = chunk_for(want, 1);
      } else if (at.n_splits < attention_max_splits()) {
        // fewer planned splits than a cluster holds (the plan rounds its chunk up to whole tiles):
        // a cluster's worth anyway; the kernel shares the step's actual context over them, so at
        // short contexts a split holds one tile instead of two (batch 1 at context ~650: 6.78 -> 6.67 ms)
        const int ns = std::min(attention_max_splits(), want);
        at.n_splits = ns;
        at.chunk = chunk_for(ns, 1);
      } else if (at.n_splits >= 2 && p.n_groups <= kMaxCtxGroups) {
        // long contexts: R clusters of 8 splits share the context, R as large as keeps every CTA at
        // 4 or more tiles of 64 positions, the clusters within what the occupancy calculator says
        // the device holds at once and the CTAs within 3/4 of the per-SM count. Measured on the
        // 16K-context step, where the calculator allows 36 clusters of 8 at two CTAs per SM: the
        // 8B verify's 32 clusters (256 CTAs, the per-SM count's 304 nearly full) still ran partly in
        // a second wave, 24 did not (4.25 -> 3.84 ms); the 1B drafter's 32 (of 608) did not (step
        // 1.02 -> 0.93 ms); clusters of 16 lost to clusters of 8 at every CTA count.
        const int ns = std::min(at.n_splits, 8);
        int best_R = 0;
        for (int Rc = 1; Rc <= kMaxCtxClusters; ++Rc) {
          const long per_head = static_cast<long>(ns) * Rc;
          if (4 * per_head * p.n_groups * Hkv > 3 * resident || max_ctx < 64 * 4 * per_head) break;
          AttnArgs t = at;
          t.n_splits = ns; t.n_ctx_clusters = Rc; t.chunk = chunk_for(ns, Rc);
          t.part_acc = c->attn_part_acc; t.part_ml = c->attn_part_ml; t.part_cnt = c->attn_part_cnt;
          // (not monotone in R: more CTAs per SM take less shared memory each)
          if (static_cast<long>(Rc) * p.n_groups * Hkv > attention_max_clusters(t)) continue;
          best_R = Rc;
        }
        if (best_R >= 2 && ns * best_R > at.n_splits) {   // else the planned single cluster
          at.n_splits = ns;
          at.n_ctx_clusters = best_R;
          at.chunk = chunk_for(ns, best_R);
          at.part_acc = c->attn_part_acc; at.part_ml = c->attn_part_ml; at.part_cnt = c->attn_part_cnt;
        }
      }
      // a single cluster per (group, KV head) whose clusters cannot all be resident at once would
      // run in two waves: fewer splits instead
      while (at.n_ctx_clusters == 1 && at.n_splits > 1 &&
             static_cast<long>(p.n_groups) * Hkv > attention_max_clusters(at)) {
        --at.n_splits;
        at.chunk = chunk_for(at.n_splits, 1);
      }
    }
    at.pre_len = p.pre_len; at.pre_stable = p.pre_stable; at.pre_fresh = p.pre_fresh; at.err = c->errw;
    double kvb = 0;
    if (c->prof && !c->h_n.empty()) {
      for (int b = 0; b < c->B; ++b) kvb += 2.0 * 2.0 * Hkv * hd * (c->h_n[b] + 16);
    }
    if (in_o)
      RUN_GEMM(go, gemm_bytes(M, d, H * hd, 8) + kvb);
    else {
      CK(timed(c, PC_ATTN, kvb, [&] { return attention(at, c->st); }));
      RUN_GEMM(go, gemm_bytes(M, d, H * hd, 8));
    }
    if (!fused)
      CK(timed(c, PC_OTHER, 0, [&] {
        return rmsnorm(c->x, nullptr, m.W(l, SD2_W_MLP_NORM), mc.norm_eps, M, d, c->a, nullptr, nullptr, 0, c->st);
      }));
    GemmArgs gu = gu_args(l);
    if (fused) consume(gu, parts);
    if (c->cfg.steering_site == 2 && o.bias) {   // per-row biases of the conditional MLP (below)
      gu.bias = c->rowbias; gu.ld_bias = F; gu.row_seq = c->row_ident;
    }
    RUN_GEMM(gu, gemm_bytes(M, 2 * F, d, 1));
    GemmArgs gd = down_args(l);
    if (fused && l + 1 < L) {
      produce(gd, m.W(l + 1, SD2_W_ATTN_NORM));
      gd.tap = o.taps; gd.tap_row = o.tap_row; gd.tap_mask = tap_mask(l + 1);
      parts = gemm_norm_parts(gd);
    } else if (fused && final_in_down) {   // the final RMSNorm of a head that takes every row
      produce(gd, m.final_norm);
      gd.tap = o.taps; gd.tap_row = o.tap_row; gd.tap_mask = tap_mask(L);
      parts = gemm_norm_parts(gd);
    }
    RUN_GEMM(gd, gemm_bytes(M, d, F, 8));
  }
  return head(c, m, p, o, fused && final_in_down ? parts : 0);
}

// a1: g = LN(W_hml [h; m; l]) at each sequence's steering row, biases = W_s g.
sd2_status steer(sd2_ctx* c, const int* row_idx) {
  const int B = c->B, dv = c->V.c.d_model, dg = c->cfg.d_steer, k = c->cfg.k;
  const int nb = c->D.c.n_layers * bias_width(c);
  CK(timed(c, PC_OTHER, 0, [&] {
    return gather_rows_bf16(c->taps, (k + 1) * 3 * dv, row_idx, 3 * dv, B, c->hml_in, c->st);
  }));
  GemmArgs g{};
  g.x = c->hml_in; g.ldx = 3 * dv; g.M = B; g.K = 3 * dv;
  g.seg[0] = {c->w_hml, dg}; g.nseg = 1; g.epi = EPI_STORE; g.out = c->g_pre; g.ldo = dg;
  RUN_GEMM(g, gemm_bytes(B, dg, 3 * dv, 4));
  CK(timed(c, PC_OTHER, 0, [&] {
    return layernorm(c->g_pre, c->ln_g, c->ln_b, c->cfg.steer_ln_eps, B, dg, c->g, c->g_bf, c->st);
  }));
  GemmArgs gs{};
  gs.x = c->g_bf; gs.ldx = dg; gs.M = B; gs.K = dg;
  if (c->cfg.steering_site == 2) {        // the g half of the conditional bias MLP's first layer
    const int ncg = c->D.c.n_layers * dg;
    gs.seg[0] = {c->w_c1g, ncg}; gs.nseg = 1; gs.epi = EPI_STORE; gs.out = c->cg; gs.ldo = ncg;
    RUN_GEMM(gs, gemm_bytes(B, ncg, dg, 4));
    return SD2_OK;
  }
  gs.seg[0] = {c->w_s, nb}; gs.nseg = 1; gs.epi = EPI_STORE; gs.out = c->bias; gs.ldo = nb;
  RUN_GEMM(gs, gemm_bytes(B, nb, dg, 4));
  return SD2_OK;
}

sd2_status run_step(sd2_ctx* c) {
  const int B = c->B, k = c->cfg.k, V = c->V.c.vocab;
  cudaEvent_t s0 = nullptr, s1 = nullptr;
  auto stage_begin = [&]() {
    if (c->prof) { s0 = take_event(c); cudaEventRecord(s0, c->st); }
  };
  auto stage_end = [&](int cls, double bytes) {
    if (c->prof) { s1 = take_event(c); cudaEventRecord(s1, c->st); c->recs.push_back({cls, bytes, s0, s1}); }
  };
  auto mark = [&](int i) {
    if (c->stage_on) cudaEventRecordWithFlags(c->stage_ev[i], c->st, cudaEventRecordExternal);
  };
  if (c->gemm_timing) {
    // every stamp slot: entry and wait times at their maximum, exit time at zero
    c->gstamp_n = 0;
    c->gstamp_bytes.clear();
    c->gstamp_stage.clear();
    CK(cudaMemset2DAsync(c->gstamp, 24, 0xFF, 16, kMaxStampedLaunches, c->st));
    CK(cudaMemset2DAsync(c->gstamp + 2, 24, 0, 8, kMaxStampedLaunches, c->st));
  }
  mark(0);
  stage_begin();
  sd2_status s = SD2_OK;
  c->cur_stage = 0;
  if (!c->cfg.no_steering && (s = steer(c, c->state + 2 * c->maxB)) != SD2_OK) return s;
  stage_end(PC_STEER, 2.0 * c->cfg.d_steer * 3 * c->V.c.d_model +
                          2.0 * c->cfg.d_steer * c->D.c.n_layers * static_cast<double>(c->D.c.d_ffn));
  mark(1);
  for (int i = 1; i <= k; ++i) {
    stage_begin();
    c->cur_stage = i;
    const Plan& p = (i == 1) ? c->p_d1 : c->p_dn;
    CK(timed(c, PC_OTHER, 0, [&] {
      return plan_rows(i == 1 ? PLAN_DRAFT_FIRST : PLAN_DRAFT_NEXT, i, B, k, c->cfg.max_ctx, c->state, c->maxB,
                       c->committed, c->xhat, c->row_tok, c->row_pos, c->row_seq, c->row_valid, c->st);
    }));
    FwdOut o;
    o.bias = c->cfg.no_steering ? nullptr : c->bias;
    o.logit_rows = (i == 1) ? c->logit_rows_d1 : nullptr;
    o.n_logit_rows = B;
    o.logits = c->logits_d + static_cast<size_t>(i - 1) * V;
    o.ld_logits = static_cast<long long>(k) * V;
    s = chain_takes(c, p) ? forward_chain(c, c->D, p, o) : forward(c, c->D, p, o);
    if (s != SD2_OK) return s;
    CK(timed(c, PC_SAMPLE, 4.0 * B * V, [&] {
      return sample_rows(o.logits, o.ld_logits, B, V, c->temp, Seed{0, c->seed_d}, RNG_DRAFT, i, c->iter, 0, c->xhat + (i - 1), k,
                         nullptr, 0, c->samp_slot, c->samp_counter, c->errw, c->st);
    }));
    stage_end(PC_DRAFT, 2.0 * c->D.c.n_layers * (static_cast<double>(c->D.c.d_model) * c->D.qkv_width() +
                                                  static_cast<double>(c->D.c.n_heads) * c->D.c.head_dim * c->D.c.d_model +
                                                  3.0 * c->D.c.d_model * c->D.c.d_ffn) +
                            2.0 * V * c->D.c.d_model);
    mark(1 + i);
  }
  stage_begin();
  c->cur_stage = k + 1;
  CK(timed(c, PC_OTHER, 0, [&] {
    return plan_rows(PLAN_VERIFY, 0, B, k, c->cfg.max_ctx, c->state, c->maxB, c->committed, c->xhat, c->row_tok,
                     c->row_pos, c->row_seq, c->row_valid, c->st);
  }));
  FwdOut o;
  o.taps = c->taps;
  o.tap_row = nullptr;
  for (int t = 0; t < 3; ++t) o.tap_layers[t] = c->cfg.tap_layers[t];
  o.n_logit_rows = B * (k + 1);
  o.logit_rows = nullptr;
  o.logits = c->logits_t;
  o.ld_logits = V;
  s = forward(c, c->V, c->p_v, o);
  if (s != SD2_OK) return s;
  stage_end(PC_VERIFY, 2.0 * c->V.c.n_layers * (static_cast<double>(c->V.c.d_model) * c->V.qkv_width() +
                                                 static_cast<double>(c->V.c.n_heads) * c->V.c.head_dim * c->V.c.d_model +
                                                 3.0 * c->V.c.d_model * c->V.c.d_ffn) +
                          2.0 * V * c->V.c.d_model);
  mark(k + 2);
  c->cur_stage = -1;
  return SD2_OK;
}

sd2_status run_accept(sd2_ctx* c) {
  const int B = c->B, k = c->cfg.k, V = c->V.c.vocab;
  CK(timed(c, PC_ACCEPT, 4.0 * B * (2 * k + 1) * V, [&] {
    return accept_blocks(c->logits_t, c->logits_d, SD2_DTYPE_F32, c->xhat, c->temp, B, k, V, Seed{0, c->seed_d}, 0, c->iter,
                         c->state + 3 * c->maxB, c->tok_out, c->n_out, c->as, c->errw, c->st);
  }));
  CK(timed(c, PC_OTHER, 0, [&] {
    return commit(B, k, c->cfg.max_ctx, c->state, c->maxB, c->committed, c->tok_out, c->n_out, c->iter, c->st);
  }));
  return SD2_OK;
}

template <typename F>
sd2_status capture(sd2_ctx* c, cudaGraphExec_t* exec, F body) {
  cudaStream_t user = c->st;
  c->st = c->cap_st;
  cudaError_t e = cudaStreamBeginCapture(c->st, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) { c->st = user; return fail(c, SD2_ECUDA, std::string("begin capture: ") + cudaGetErrorString(e)); }
  sd2_status s = body();
  cudaGraph_t graph = nullptr;
  e = cudaStreamEndCapture(c->st, &graph);
  c->st = user;
  if (s != SD2_OK) { if (graph) cudaGraphDestroy(graph); return s; }
  if (e != cudaSuccess) return fail(c, SD2_ECUDA, std::string("end capture: ") + cudaGetErrorString(e));
  e = cudaGraphInstantiate(exec, graph, 0);
  cudaGraphDestroy(graph);
  if (e != cudaSuccess) return fail(c, SD2_ECUDA, std::string("graph instantiate: ") + cudaGetErrorString(e));
  return SD2_OK;
}

void drop_graphs(sd2_ctx* c) {
  if (c->g_step) cudaGraphExecDestroy(c->g_step);
  if (c->g_accept) cudaGraphExecDestroy(c->g_accept);
  c->g_step = c->g_accept = nullptr;
}

// Context positions per attention split: whole 64-position tiles, at most attention_max_splits()
// splits (one cluster).
int attn_chunk(int max_ctx) {
  const int span = 64 * attention_max_splits();
  return 64 * std::max(1, (max_ctx + span - 1) / span);
}

// Attention row groups: consecutive rows of one sequence, at most `cap` rows per group.
void add_groups(std::vector<int>& r0, std::vector<int>& nr, std::vector<int>& sq, int row0, int rows, int seq, int cap) {
  for (int t = 0; t < rows; t += cap) {
    r0.push_back(row0 + t);
    nr.push_back(std::min(cap, rows - t));
    sq.push_back(seq);
  }
}

}  // namespace

namespace sd2 {
// Sets the text sd2_last_error(NULL) returns, for context-free entry points in other files.
void record_last_error(const std::string& m) { g_last_error = m; }
}  // namespace sd2

// ------------------------------------------------------------------------------------------------
// C ABI
// ------------------------------------------------------------------------------------------------
extern "C" {

const char* sd2_last_error(const sd2_ctx* c) { return c ? c->err.c_str() : g_last_error.c_str(); }

sd2_status sd2_init(const sd2_config* cfg, const sd2_weights* w, void* stream, sd2_ctx** out) {
  sd2_ctx* c = nullptr;
  if (!cfg || !w || !out) return fail(nullptr, SD2_EINVAL, "null argument");
  *out = nullptr;
  if (!valid_lm(cfg->verifier) || !valid_lm(cfg->drafter))
    return fail(nullptr, SD2_EINVAL, "unsupported model shape (head_dim 64/128, dims multiple of 8, vocab of 4)");
  if (cfg->verifier.vocab != cfg->drafter.vocab) return fail(nullptr, SD2_EINVAL, "verifier and drafter vocab differ");
  if (cfg->k < 1 || cfg->k > 16) return fail(nullptr, SD2_EINVAL, "k must be in [1, 16]");
  if (cfg->max_batch < 1 || cfg->max_batch > 256) return fail(nullptr, SD2_EINVAL, "max_batch must be in [1, 256]");
  if (cfg->kv_block != 16) return fail(nullptr, SD2_EINVAL, "kv_block must be 16");
  if (cfg->max_ctx < cfg->k + 3) return fail(nullptr, SD2_EINVAL, "max_ctx too small for one block");
  if (cfg->d_steer <= 0 || cfg->d_steer % 8) return fail(nullptr, SD2_EINVAL, "d_steer must be a positive multiple of 8");
  if (cfg->max_prefill_tokens < 1) return fail(nullptr, SD2_EINVAL, "max_prefill_tokens must be positive");
  if (cfg->steering_site < 0 || cfg->steering_site > 2) return fail(nullptr, SD2_EINVAL, "steering_site must be 0, 1 or 2");
  for (int t = 0; t < 3; ++t)
    if (cfg->tap_layers[t] < 1 || cfg->tap_layers[t] > cfg->verifier.n_layers)
      return fail(nullptr, SD2_EINVAL, "tap_layers must be 1-based verifier layers");
  if (!cfg->no_steering && (!aligned16(w->w_hml) || !w->steer_ln_gamma || !w->steer_ln_beta ||
                            (cfg->steering_site == 2 ? !aligned16(w->w_c1x) || !aligned16(w->w_c1g) || !aligned16(w->w_c2)
                                                     : !aligned16(w->w_s))))
    return fail(nullptr, SD2_EINVAL, "steering weights null or not 16-byte aligned");

  c = new sd2_ctx();
  c->cfg = *cfg;
  c->st = static_cast<cudaStream_t>(stream);
  c->maxB = cfg->max_batch;
  c->w_hml = w->w_hml; c->ln_g = w->steer_ln_gamma; c->ln_b = w->steer_ln_beta; c->w_s = w->w_s;
  c->w_c1x = w->w_c1x; c->w_c1g = w->w_c1g; c->w_c2 = w->w_c2;
  sd2_status s;
  if ((s = load_model(c, c->V, cfg->verifier, w->verifier, "verifier")) != SD2_OK ||
      (s = load_model(c, c->D, cfg->drafter, w->drafter, "drafter")) != SD2_OK) {
    g_last_error = c->err;
    sd2_free(c);
    return s;
  }
  const int k = cfg->k, maxB = c->maxB, Vv = cfg->verifier.vocab;
  const int step_rows = std::max(maxB * (k + 1), 2 * maxB);
  c->max_rows = std::max(cfg->max_prefill_tokens, step_rows);
  const int R = c->max_rows;
  const int dmax = std::max(cfg->verifier.d_model, cfg->drafter.d_model);
  const int fmax = std::max(cfg->verifier.d_ffn, cfg->drafter.d_ffn);
  const int qkvmax = std::max(c->V.qkv_width(), c->D.qkv_width());
  const int hmax = std::max(cfg->verifier.n_heads * cfg->verifier.head_dim, cfg->drafter.n_heads * cfg->drafter.head_dim);
  auto go = [&]() -> sd2_status {
    ALLOC(c->state, 4 * maxB);
    ALLOC(c->committed, static_cast<size_t>(maxB) * cfg->max_ctx);
    ALLOC(c->iter, 1);
    ALLOC(c->seed_d, 1);
    ALLOC(c->xhat, static_cast<size_t>(maxB) * k);
    ALLOC(c->temp, maxB);
    ALLOC(c->errw, 1);
    ALLOC(c->row_tok, R); ALLOC(c->row_pos, R); ALLOC(c->row_seq, R); ALLOC(c->row_valid, R);
    c->statics_cap = 8 * R + 64;
    ALLOC(c->statics, c->statics_cap);
    ALLOC(c->x, static_cast<size_t>(R) * dmax);
    ALLOC(c->a, static_cast<size_t>(R) * dmax * 2);
    ALLOC(c->qkv, static_cast<size_t>(R) * qkvmax);
    ALLOC(c->q, static_cast<size_t>(R) * hmax);
    ALLOC(c->attn, static_cast<size_t>(R) * hmax * 2);
    {
      // [kMaxCtxGroups][Hkv][kMaxCtxClusters][64 * 128 / 4] float4 + float2 partials,
      // [kMaxCtxGroups][Hkv][16] counters
      const int hkv = std::max(cfg->verifier.n_kv_heads, cfg->drafter.n_kv_heads);
      const size_t slots = static_cast<size_t>(kMaxCtxGroups) * hkv * kMaxCtxClusters * 64 * 32;
      ALLOC(c->attn_part_acc, slots * 16);
      ALLOC(c->attn_part_ml, slots * 8);
      ALLOC(c->attn_part_cnt, static_cast<size_t>(kMaxCtxGroups) * hkv * 16 * 4);
      CK(cudaMemset(c->attn_part_cnt, 0, static_cast<size_t>(kMaxCtxGroups) * hkv * 16 * 4));
      // flat-mode attention: a slot per resident CTA of either model ([Hkv][W][64][hd] f32 and
      // [Hkv][W][64] float2, W * Hkv <= the resident CTAs), counters [kMaxFlatGroups][Hkv]
      size_t acc_b = 0, ml_b = 0;
      for (const sd2_lm_config* mc : {&cfg->verifier, &cfg->drafter}) {
        const size_t ctas = static_cast<size_t>(attention_ctas_per_sm(mc->head_dim)) * sm_count_cached();
        acc_b = std::max(acc_b, ctas * 64 * mc->head_dim * 4);
        ml_b = std::max(ml_b, ctas * 64 * 8);
      }
      ALLOC(c->attn_flat_acc, acc_b);
      ALLOC(c->attn_flat_ml, ml_b);
      ALLOC(c->attn_flat_cnt, static_cast<size_t>(kMaxFlatGroups) * hkv);
      CK(cudaMemset(c->attn_flat_cnt, 0, static_cast<size_t>(kMaxFlatGroups) * hkv * sizeof(unsigned)));
    }
    ALLOC(c->h, static_cast<size_t>(R) * fmax * 2);
    ALLOC(c->ssq, static_cast<size_t>(R) * (dmax / 128 + 1) * 8);
    if (cfg->steering_site == 2) {
      const int Ld = cfg->drafter.n_layers, dd = cfg->drafter.d_model, dg = cfg->d_steer;
      ALLOC(c->cg, static_cast<size_t>(maxB) * Ld * dg);
      ALLOC(c->fb, static_cast<size_t>(R) * dd * 2);      // bf16 (void buffers are sized in bytes)
      ALLOC(c->cu_h, static_cast<size_t>(R) * dg * 2);
      ALLOC(c->rowbias, static_cast<size_t>(R) * cfg->drafter.d_ffn);
      ALLOC(c->row_ident, R);
      std::vector<int> ident(R);
      for (int i = 0; i < R; ++i) ident[i] = i;
      CK(cudaMemcpy(c->row_ident, ident.data(), sizeof(int) * R, cudaMemcpyHostToDevice));
    }
    ALLOC(c->logits_t, static_cast<size_t>(maxB) * (k + 1) * Vv);
    ALLOC(c->logits_d, static_cast<size_t>(maxB) * k * Vv);
    ALLOC(c->taps, static_cast<size_t>(maxB) * (k + 1) * 3 * cfg->verifier.d_model);
    ALLOC(c->hml_in, static_cast<size_t>(maxB) * 3 * cfg->verifier.d_model * 2);
    ALLOC(c->g_pre, static_cast<size_t>(maxB) * cfg->d_steer);
    ALLOC(c->g, static_cast<size_t>(maxB) * cfg->d_steer);
    ALLOC(c->g_bf, static_cast<size_t>(maxB) * cfg->d_steer * 2);
    ALLOC(c->bias, static_cast<size_t>(maxB) * cfg->drafter.n_layers *
                       std::max(cfg->drafter.d_ffn, cfg->drafter.d_model));
    ALLOC(c->samp_slot, maxB);
    ALLOC(c->samp_counter, maxB);
    void* acc;
    ALLOC(acc, accept_scratch_bytes(maxB, k));
    c->as = accept_scratch_carve(acc, maxB, k);
    ALLOC(c->tok_out, static_cast<size_t>(maxB) * (k + 1));
    ALLOC(c->n_out, maxB);
    ALLOC(c->first, maxB);
    ALLOC(c->cu, maxB + 1);
    ALLOC(c->gen_prompt, cfg->max_prefill_tokens);
    ALLOC(c->gen_first, maxB);
    ALLOC(c->gen_tok, static_cast<size_t>(maxB) * (k + 1));
    ALLOC(c->gen_n, maxB);
    if (cudaHostAlloc(reinterpret_cast<void**>(&c->gen_host), sizeof(int) * static_cast<size_t>(maxB) * (k + 2),
                      cudaHostAllocDefault) != cudaSuccess) {
      cudaGetLastError();
      c->gen_host = nullptr;
      return fail(c, SD2_ENOMEM, "cudaHostAlloc of the pinned token staging buffer failed");
    }
    CK(cudaMemset(c->samp_slot, 0, sizeof(unsigned long long) * maxB));
    CK(cudaMemset(c->samp_counter, 0, sizeof(int) * maxB));
    CK(cudaMemset(c->errw, 0, sizeof(unsigned)));
    CK(cudaMemset(c->state, 0, sizeof(int) * 4 * maxB));
    CK(cudaMemset(c->taps, 0, sizeof(float) * static_cast<size_t>(maxB) * (k + 1) * 3 * cfg->verifier.d_model));
    CK(cudaStreamCreateWithFlags(&c->cap_st, cudaStreamNonBlocking));
    // the drafter's persistent layer chain, when its shape allows (the step plans stay within it)
    const sd2_lm_config& dc = cfg->drafter;
    if (chain_plan(c->chain, dc.n_layers, dc.d_model, dc.n_heads, dc.n_kv_heads, dc.head_dim, dc.d_ffn, dc.vocab,
                   dc.norm_eps, attention_max_splits())) {
      unsigned char* block;
      ALLOC(block, chain_device_bytes(c->chain));
      CK(chain_prepare(c->chain, c->D.w.data(), c->D.embed, c->D.cache(), c->D.rope_cs, block));
      c->chain_ok = true;
    }
    return SD2_OK;
  };
  if ((s = go()) != SD2_OK) {
    g_last_error = c->err;
    sd2_free(c);
    return s;
  }
  *out = c;
  return SD2_OK;
}

sd2_status sd2_prefill(sd2_ctx* c, int32_t batch, const int32_t* d_tokens, const int32_t* h_cu_lens,
                       const float* h_temperature, uint64_t seed, int32_t* d_first_token) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  if (!d_tokens || !h_cu_lens || !h_temperature) return fail(c, SD2_EINVAL, "null argument");
  if (batch < 1 || batch > c->maxB) return fail(c, SD2_ECAPACITY, "batch exceeds max_batch");
  const int k = c->cfg.k, V = c->V.c.vocab;
  if (h_cu_lens[0] != 0) return fail(c, SD2_EINVAL, "h_cu_lens[0] must be 0");
  int total = 0, maxlen = 0;
  for (int b = 0; b < batch; ++b) {
    const int len = h_cu_lens[b + 1] - h_cu_lens[b];
    if (len < 1) return fail(c, SD2_EINVAL, "empty prompt");
    if (len + k + 2 > c->cfg.max_ctx) return fail(c, SD2_ECAPACITY, "prompt too long for max_ctx");
    if (!(h_temperature[b] >= 0.f) || !isfinite(h_temperature[b])) return fail(c, SD2_EINVAL, "bad temperature");
    total += len;
    maxlen = std::max(maxlen, len);
  }
  if (total > c->cfg.max_prefill_tokens) return fail(c, SD2_ECAPACITY, "prompt tokens exceed max_prefill_tokens");
  c->B = batch;
  c->seed = seed;
  c->phase = 0;

  // host-built plans: prefill rows, then the static groups of the step shapes
  std::vector<int> pos(total), seq(total), valid(total, 1), logit_rows(batch), tap_row(total, -1);
  for (int b = 0; b < batch; ++b) {
    for (int t = h_cu_lens[b]; t < h_cu_lens[b + 1]; ++t) { pos[t] = t - h_cu_lens[b]; seq[t] = b; }
    logit_rows[b] = h_cu_lens[b + 1] - 1;
    tap_row[h_cu_lens[b + 1] - 1] = b * (k + 1);
  }
  std::vector<int> st;  // the statics buffer, assembled in order
  auto push = [&](const std::vector<int>& v) { int off = (int)st.size(); st.insert(st.end(), v.begin(), v.end()); return off; };
  auto groups_of = [&](const Model& m, std::vector<int>& r0, std::vector<int>& nr, std::vector<int>& sq, bool prefill) {
    const int cap = m.group_rows();
    for (int b = 0; b < batch; ++b) {
      if (prefill) add_groups(r0, nr, sq, h_cu_lens[b], h_cu_lens[b + 1] - h_cu_lens[b], b, cap);
    }
  };
  std::vector<int> vr0, vnr, vsq, dr0, dnr, dsq, d1r0, d1nr, d1sq, dnr0, dnnr, dnsq, sr0, snr, ssq, lr1;
  groups_of(c->V, vr0, vnr, vsq, true);
  groups_of(c->D, dr0, dnr, dsq, true);
  for (int b = 0; b < batch; ++b) {
    add_groups(d1r0, d1nr, d1sq, 2 * b, 2, b, c->D.group_rows());
    add_groups(dnr0, dnnr, dnsq, b, 1, b, c->D.group_rows());
    add_groups(sr0, snr, ssq, b * (k + 1), k + 1, b, c->V.group_rows());
    lr1.push_back(2 * b + 1);
  }
  // The step-shape tables come first: they depend on the batch and k alone, so a step graph captured
  // after an earlier prefill of the same batch size reads the same addresses and stays valid.
  const int o_d1r0 = push(d1r0), o_d1nr = push(d1nr), o_d1sq = push(d1sq);
  const int o_dnr0 = push(dnr0), o_dnnr = push(dnnr), o_dnsq = push(dnsq);
  const int o_sr0 = push(sr0), o_snr = push(snr), o_ssq = push(ssq), o_lr1 = push(lr1);
  std::vector<int> key = {batch, k};
  key.insert(key.end(), st.begin(), st.end());
  if (key != c->graph_key) {
    drop_graphs(c);
    c->graph_key = key;
  }
  const int o_pos = push(pos), o_seq = push(seq), o_valid = push(valid), o_lr = push(logit_rows), o_tr = push(tap_row);
  const int o_vr0 = push(vr0), o_vnr = push(vnr), o_vsq = push(vsq);
  const int o_dr0 = push(dr0), o_dnr = push(dnr), o_dsq = push(dsq);
  std::vector<int> cu(h_cu_lens, h_cu_lens + batch + 1);
  const int o_cu = push(cu);
  if ((int)st.size() > c->statics_cap) {
    drop_graphs(c);
    c->graph_key.clear();
    return fail(c, SD2_ECAPACITY, "plan tables exceed their buffer");
  }
  CK(cudaMemcpyAsync(c->statics, st.data(), st.size() * sizeof(int), cudaMemcpyHostToDevice, c->st));
  CK(cudaMemcpyAsync(c->seed_d, &seed, sizeof(seed), cudaMemcpyHostToDevice, c->st));
  std::vector<float> temps(h_temperature, h_temperature + batch);
  CK(cudaMemcpyAsync(c->temp, temps.data(), batch * sizeof(float), cudaMemcpyHostToDevice, c->st));
  CK(cudaMemsetAsync(c->iter, 0, sizeof(int), c->st));
  const int* S = c->statics;
  Plan pv;
  pv.M = total; pv.tok = d_tokens; pv.pos = S + o_pos; pv.seq = S + o_seq; pv.valid = S + o_valid;
  pv.n_groups = (int)vr0.size(); pv.g_row0 = S + o_vr0; pv.g_nrows = S + o_vnr; pv.g_seq = S + o_vsq;
  pv.n_splits = 1; pv.chunk = ((maxlen + 63) / 64) * 64; pv.max_rows = std::min(maxlen, c->V.group_rows());
  Plan pd = pv;
  pd.n_groups = (int)dr0.size(); pd.g_row0 = S + o_dr0; pd.g_nrows = S + o_dnr; pd.g_seq = S + o_dsq;
  pd.max_rows = std::min(maxlen, c->D.group_rows());
  // step-shape plans (rows filled on the device each step)
  const int chunk = attn_chunk(c->cfg.max_ctx), splits = (c->cfg.max_ctx + chunk - 1) / chunk;
  auto step_plan = [&](int M, int ng, int o0, int o1, int o2, int rows) {
    Plan p;
    p.max_rows = rows;
    p.M = M; p.tok = c->row_tok; p.pos = c->row_pos; p.seq = c->row_seq; p.valid = c->row_valid;
    p.n_groups = ng; p.g_row0 = S + o0; p.g_nrows = S + o1; p.g_seq = S + o2; p.n_splits = splits; p.chunk = chunk;
    return p;
  };
  c->p_d1 = step_plan(2 * batch, (int)d1r0.size(), o_d1r0, o_d1nr, o_d1sq, std::min(2, c->D.group_rows()));
  c->p_dn = step_plan(batch, (int)dnr0.size(), o_dnr0, o_dnnr, o_dnsq, 1);
  c->p_v = step_plan(batch * (k + 1), (int)sr0.size(), o_sr0, o_snr, o_ssq, std::min(k + 1, c->V.group_rows()));
  // State rows written before each step (by the previous commit or the prefill): the drafter cache
  // holds positions [0, D), the verifier cache [0, n - 1). A drafter step's rows lie in [D, D + k + 1)
  // (at most 2 pending tokens, then the drafts), the verify rows in [n - 1, n + k).
  c->p_d1.pre_len = c->p_dn.pre_len = c->state + c->maxB;
  c->p_d1.pre_fresh = c->p_dn.pre_fresh = k + 1;
  c->p_v.pre_len = c->state;
  c->p_v.pre_stable = -1;
  c->p_v.pre_fresh = k + 1;
  c->logit_rows_d1 = S + o_lr1;

  // verifier over the prompts: logits of each last row -> row b*(k+1) of the target buffer
  FwdOut o;
  o.taps = c->taps; o.tap_row = S + o_tr;
  for (int t = 0; t < 3; ++t) o.tap_layers[t] = c->cfg.tap_layers[t];
  o.logit_rows = S + o_lr; o.n_logit_rows = batch; o.logits = c->logits_t; o.ld_logits = static_cast<long long>(k + 1) * V;
  sd2_status s = forward(c, c->V, pv, o);
  if (s != SD2_OK) return s;
  CK(sample_rows(c->logits_t, static_cast<long long>(k + 1) * V, batch, V, c->temp, Seed{seed, nullptr}, RNG_RESAMPLE, 0, nullptr, 0,
                 c->first, 1, nullptr, 0, c->samp_slot, c->samp_counter, c->errw, c->st));
  CK(prefill_init(batch, c->cfg.max_ctx, d_tokens, S + o_cu, c->first, c->state, c->maxB, c->committed, d_first_token,
                  c->st));
  // steering from the last prompt row (j = 0 -> tap row b*(k+1)), then the drafter prefill
  if (!c->cfg.no_steering && (s = steer(c, c->state + 2 * c->maxB)) != SD2_OK) return s;
  FwdOut od;
  od.bias = c->cfg.no_steering ? nullptr : c->bias;
  s = forward(c, c->D, pd, od);
  if (s != SD2_OK) return s;
  const int one = 1;
  CK(cudaMemcpyAsync(c->iter, &one, sizeof(int), cudaMemcpyHostToDevice, c->st));
  CK(cudaStreamSynchronize(c->st));  // host staging buffers above go out of scope
  c->phase = 1;
  return SD2_OK;
}

sd2_status sd2_step(sd2_ctx* c) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  if (c->phase != 1) return fail(c, SD2_ESTATE, "sd2_step needs a prefill or an accepted previous step");
  if (c->prof) {
    c->h_n.assign(c->B, 0);
    CK(cudaMemcpyAsync(c->h_n.data(), c->state, sizeof(int) * c->B, cudaMemcpyDeviceToHost, c->st));
    CK(cudaStreamSynchronize(c->st));
  }
  sd2_status s;
  if (c->use_graphs && !c->prof) {
    if (!c->g_step && (s = capture(c, &c->g_step, [&] { return run_step(c); })) != SD2_OK) return s;
    CK(cudaGraphLaunch(c->g_step, c->st));
  } else if ((s = run_step(c)) != SD2_OK) {
    return s;
  }
  if (c->stage_on) c->stage_done = true;
  if (c->gemm_timing) c->gemm_timing_done = true;
  c->phase = 2;
  return SD2_OK;
}

sd2_status sd2_accept(sd2_ctx* c, int32_t* d_tokens, int32_t* d_n) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  if (c->phase != 2) return fail(c, SD2_ESTATE, "sd2_accept needs a preceding sd2_step");
  if (!d_tokens || !d_n) return fail(c, SD2_EINVAL, "null output");
  sd2_status s;
  if (c->use_graphs && !c->prof) {
    if (!c->g_accept && (s = capture(c, &c->g_accept, [&] { return run_accept(c); })) != SD2_OK) return s;
    CK(cudaGraphLaunch(c->g_accept, c->st));
  } else if ((s = run_accept(c)) != SD2_OK) {
    return s;
  }
  CK(cudaMemcpyAsync(d_tokens, c->tok_out, sizeof(int) * c->B * (c->cfg.k + 1), cudaMemcpyDeviceToDevice, c->st));
  CK(cudaMemcpyAsync(d_n, c->n_out, sizeof(int) * c->B, cudaMemcpyDeviceToDevice, c->st));
  c->phase = 1;
  return SD2_OK;
}

sd2_status sd2_generate(sd2_ctx* c, int32_t batch, const int32_t* h_tokens, const int32_t* h_cu_lens,
                        const float* h_temperature, uint64_t seed, int32_t max_new, int32_t* h_out, int32_t* h_n_out) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  if (!h_tokens || !h_cu_lens || !h_temperature || !h_out || !h_n_out) return fail(c, SD2_EINVAL, "null argument");
  if (batch < 1 || batch > c->maxB) return fail(c, SD2_ECAPACITY, "batch exceeds max_batch");
  if (max_new < 1) return fail(c, SD2_EINVAL, "max_new must be positive");
  if (h_cu_lens[0] != 0 || h_cu_lens[batch] < batch) return fail(c, SD2_EINVAL, "bad h_cu_lens");
  const int total = h_cu_lens[batch], k = c->cfg.k;
  if (total > c->cfg.max_prefill_tokens) return fail(c, SD2_ECAPACITY, "prompt tokens exceed max_prefill_tokens");
  CK(cudaMemcpyAsync(c->gen_prompt, h_tokens, sizeof(int) * static_cast<size_t>(total), cudaMemcpyHostToDevice, c->st));
  sd2_status s = sd2_prefill(c, batch, c->gen_prompt, h_cu_lens, h_temperature, seed, c->gen_first);
  if (s != SD2_OK) return s;
  int* host = c->gen_host;
  CK(cudaMemcpyAsync(host, c->gen_first, sizeof(int) * batch, cudaMemcpyDeviceToHost, c->st));
  CK(cudaStreamSynchronize(c->st));
  std::vector<char> stopped(batch, 0);
  for (int b = 0; b < batch; ++b) {
    h_out[static_cast<size_t>(b) * max_new] = host[b];
    h_n_out[b] = 1;
  }
  for (;;) {
    bool more = false;
    for (int b = 0; b < batch; ++b) more |= !stopped[b] && h_n_out[b] < max_new;
    if (!more) break;
    if ((s = sd2_step(c)) != SD2_OK) return s;
    if ((s = sd2_accept(c, c->gen_tok, c->gen_n)) != SD2_OK) return s;
    CK(cudaMemcpyAsync(host, c->gen_tok, sizeof(int) * batch * (k + 1), cudaMemcpyDeviceToHost, c->st));
    CK(cudaMemcpyAsync(host + static_cast<size_t>(batch) * (k + 1), c->gen_n, sizeof(int) * batch,
                       cudaMemcpyDeviceToHost, c->st));
    CK(cudaStreamSynchronize(c->st));
    const int* hn = host + static_cast<size_t>(batch) * (k + 1);
    for (int b = 0; b < batch; ++b) {
      if (hn[b] <= 0) { stopped[b] = 1; continue; }      // capacity reached: the sequence has stopped
      for (int t = 0; t < hn[b] && h_n_out[b] < max_new; ++t)
        h_out[static_cast<size_t>(b) * max_new + h_n_out[b]++] = host[b * (k + 1) + t];
    }
  }
  return SD2_OK;
}

sd2_status sd2_check(sd2_ctx* c) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  unsigned w = 0;
  CK(cudaStreamSynchronize(c->st));
  CK(cudaMemcpy(&w, c->errw, sizeof(unsigned), cudaMemcpyDeviceToHost));
  CK(cudaMemset(c->errw, 0, sizeof(unsigned)));
  if (w & ERR_NONFINITE) return fail(c, SD2_ENUMERIC, "non-finite logits seen on the device");
  if (w & ERR_TIMEOUT) return fail(c, SD2_ETIMEOUT, "a device-side wait timed out");
  if (w & ERR_RANGE) return fail(c, SD2_ECAPACITY, "an attention row lay outside the positions planned for the step");
  return SD2_OK;
}

sd2_status sd2_debug_fail_alloc(int32_t after) {
  g_fail_alloc_after.store(after < 0 ? -1 : after);
  return SD2_OK;
}

sd2_status sd2_debug_expire_wait(sd2_ctx* c, int64_t cycles) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  if (cycles < 1 || cycles > sd2::tc::kWaitCycles) return fail(c, SD2_EINVAL, "cycles must be in [1, the kernels' wait budget]");
  CK(expire_wait(c->errw, cycles, c->st));
  return SD2_OK;
}

sd2_status sd2_set_graphs(sd2_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  c->use_graphs = enable != 0;
  if (!c->use_graphs) drop_graphs(c);
  return SD2_OK;
}

sd2_status sd2_set_gemm_impl(sd2_ctx* c, int32_t impl) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  if (impl != 0 && impl != 1) return fail(c, SD2_EINVAL, "impl must be 0 (tensor cores) or 1 (CUDA cores)");
  c->gemm_impl = impl;
  drop_graphs(c);
  return SD2_OK;
}

sd2_status sd2_set_fused_attention(sd2_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  c->attn_in_o = enable != 0;
  drop_graphs(c);
  return SD2_OK;
}

sd2_status sd2_set_drafter_chain(sd2_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  c->use_chain = enable != 0;
  drop_graphs(c);
  return SD2_OK;
}

sd2_status sd2_free(sd2_ctx* c) {
  if (!c) return SD2_OK;
  if (c->st) cudaStreamSynchronize(c->st);
  drop_graphs(c);
  for (void* p : c->allocs) cudaFree(p);
  for (auto& r : c->recs) { cudaEventDestroy(r.e0); cudaEventDestroy(r.e1); }
  for (auto e : c->ev_pool) cudaEventDestroy(e);
  for (auto e : c->stage_ev)
    if (e) cudaEventDestroy(e);
  if (c->cap_st) cudaStreamDestroy(c->cap_st);
  if (c->gen_host) cudaFreeHost(c->gen_host);
  delete c;
  return SD2_OK;
}

sd2_status sd2_debug_buffer(const sd2_ctx* c, int32_t which, void** d_ptr, int64_t* n_elems, int32_t* dtype) {
  if (!c || !d_ptr || !n_elems || !dtype) return fail(nullptr, SD2_EINVAL, "null argument");
  const int64_t B = c->B, k = c->cfg.k, V = c->V.c.vocab;
  switch (which) {
    case 0: *d_ptr = c->logits_t; *n_elems = B * (k + 1) * V; *dtype = SD2_DTYPE_F32; break;
    case 1: *d_ptr = c->logits_d; *n_elems = B * k * V; *dtype = SD2_DTYPE_F32; break;
    case 2: *d_ptr = c->xhat; *n_elems = B * k; *dtype = -1; break;
    case 3: *d_ptr = c->taps; *n_elems = B * (k + 1) * 3 * c->V.c.d_model; *dtype = SD2_DTYPE_F32; break;
    case 4: *d_ptr = c->g; *n_elems = B * c->cfg.d_steer; *dtype = SD2_DTYPE_F32; break;
    case 5: *d_ptr = c->bias; *n_elems = B * c->D.c.n_layers * bias_width(c); *dtype = SD2_DTYPE_F32; break;
    case 6: *d_ptr = c->committed; *n_elems = B * c->cfg.max_ctx; *dtype = -1; break;
    case 7: *d_ptr = c->state; *n_elems = 4 * static_cast<int64_t>(c->maxB); *dtype = -1; break;
    case 8: *d_ptr = c->iter; *n_elems = 1; *dtype = -1; break;
    default: return fail(const_cast<sd2_ctx*>(c), SD2_EINVAL, "unknown buffer");
  }
  return SD2_OK;
}

sd2_status sd2_profile(sd2_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  c->prof = enable != 0;
  for (auto& r : c->recs) { c->ev_pool.push_back(r.e0); c->ev_pool.push_back(r.e1); }
  c->recs.clear();
  return SD2_OK;
}

sd2_status sd2_stage_timing(sd2_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  const bool on = enable != 0;
  if (on && c->stage_ev.empty()) {
    c->stage_ev.resize(c->cfg.k + 3, nullptr);
    for (auto& e : c->stage_ev) CK(cudaEventCreate(&e));
  }
  if (on != c->stage_on) drop_graphs(c);
  c->stage_on = on;
  c->stage_done = false;
  return SD2_OK;
}

sd2_status sd2_stage_read(sd2_ctx* c, double* ms) {
  if (!c || !ms) return fail(c, SD2_EINVAL, "null argument");
  if (!c->stage_on || !c->stage_done) return fail(c, SD2_ESTATE, "no step has run with stage timing on");
  CK(cudaStreamSynchronize(c->st));
  const int k = c->cfg.k;
  float t = 0;
  CK(cudaEventElapsedTime(&t, c->stage_ev[0], c->stage_ev[1]));
  ms[0] = t;
  CK(cudaEventElapsedTime(&t, c->stage_ev[1], c->stage_ev[k + 1]));
  ms[1] = t;
  CK(cudaEventElapsedTime(&t, c->stage_ev[k + 1], c->stage_ev[k + 2]));
  ms[2] = t;
  return SD2_OK;
}

sd2_status sd2_gemm_timing(sd2_ctx* c, int32_t enable) {
  if (!c) return fail(nullptr, SD2_EINVAL, "null context");
  const bool on = enable != 0;
  if (on && !c->gstamp) ALLOC(c->gstamp, 3 * static_cast<size_t>(kMaxStampedLaunches));
  if (on != c->gemm_timing) drop_graphs(c);
  c->gemm_timing = on;
  c->gemm_timing_done = false;
  return SD2_OK;
}

sd2_status sd2_gemm_timing_read(sd2_ctx* c, int32_t cap, int32_t* n, uint64_t* stamps, double* bytes, int32_t* stage) {
  if (!c || !n || !stamps || !bytes || !stage) return fail(c, SD2_EINVAL, "null argument");
  if (!c->gemm_timing || !c->gemm_timing_done) return fail(c, SD2_ESTATE, "no step has run with GEMM timing on");
  const int m = std::min(c->gstamp_n, std::max(0, cap));
  *n = c->gstamp_n;
  CK(cudaStreamSynchronize(c->st));
  if (m > 0) CK(cudaMemcpy(stamps, c->gstamp, sizeof(uint64_t) * 3 * m, cudaMemcpyDeviceToHost));
  for (int i = 0; i < m; ++i) {
    bytes[i] = c->gstamp_bytes[i];
    stage[i] = c->gstamp_stage[i];
  }
  return SD2_OK;
}

sd2_status sd2_profile_read(sd2_ctx* c, int64_t* launches, double* ms, double* bytes, int32_t n_classes) {
  if (!c || !launches || !ms || !bytes) return fail(nullptr, SD2_EINVAL, "null argument");
  CK(cudaStreamSynchronize(c->st));
  for (int i = 0; i < n_classes; ++i) { launches[i] = 0; ms[i] = 0; bytes[i] = 0; }
  for (auto& r : c->recs) {
    if (r.cls >= n_classes) continue;
    float t = 0;
    CK(cudaEventElapsedTime(&t, r.e0, r.e1));
    launches[r.cls] += 1;
    ms[r.cls] += t;
    bytes[r.cls] += r.bytes;
  }
  return SD2_OK;
}

// ------------------------------------------------------------------------------------------------
// standalone kernels
// ------------------------------------------------------------------------------------------------
size_t sd2_accept_workspace_bytes(int32_t B, int32_t k) {
  if (B < 1 || k < 1) return 0;
  return (accept_scratch_bytes(B, k) + 255) / 256 * 256;
}

sd2_status sd2_accept_logits(const void* d_target, const void* d_draft, int32_t dtype, const int32_t* d_xhat,
                             const float* d_temperature, int32_t B, int32_t k, int32_t V, uint64_t seed, uint32_t step,
                             int32_t* d_tokens, int32_t* d_n, void* d_workspace, size_t workspace_bytes, void* stream) {
  sd2_ctx* c = nullptr;
  if (!d_target || !d_draft || !d_xhat || !d_temperature || !d_tokens || !d_n || !d_workspace)
    return fail(nullptr, SD2_EINVAL, "null argument");
  if (dtype != SD2_DTYPE_F32 && dtype != SD2_DTYPE_BF16) return fail(nullptr, SD2_EINVAL, "dtype must be F32 or BF16");
  if (B < 1 || k < 1 || k > 64 || V < 4 || V % 4) return fail(nullptr, SD2_EINVAL, "need B >= 1, 1 <= k <= 64, V % 4 == 0");
  if (workspace_bytes < sd2_accept_workspace_bytes(B, k)) return fail(nullptr, SD2_EINVAL, "workspace too small");
  if (reinterpret_cast<uintptr_t>(d_workspace) & 255) return fail(nullptr, SD2_EINVAL, "workspace not 256-byte aligned");
  const size_t align = dtype == SD2_DTYPE_F32 ? 16 : 8;
  if ((reinterpret_cast<uintptr_t>(d_target) | reinterpret_cast<uintptr_t>(d_draft)) & (align - 1))
    return fail(nullptr, SD2_EINVAL, "logits not aligned for vector loads");
  unsigned* err = nullptr;
  AcceptScratch s = accept_scratch_carve(d_workspace, B, k);
  err = reinterpret_cast<unsigned*>(s.jmode + 2 * B);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  CK(cudaMemsetAsync(err, 0, sizeof(unsigned), st));
  CK(accept_blocks(d_target, d_draft, dtype, d_xhat, d_temperature, B, k, V, Seed{seed, nullptr}, step, nullptr, nullptr, d_tokens, d_n,
                   s, err, st));
  return SD2_OK;
}

size_t sd2_steer_workspace_bytes(int32_t B, int32_t d_v, int32_t d_g) {
  if (B < 1 || d_v < 1 || d_g < 1) return 0;
  const size_t b = static_cast<size_t>(B);
  // bf16 taps, f32 pre-norm g, bf16 g, and the wait flag of the tensor-core GEMMs
  return ((b * 3 * d_v * 2 + 255) / 256 + (b * d_g * 4 + 255) / 256 + (b * d_g * 2 + 255) / 256 + 1) * 256;
}

sd2_status sd2_steer(const float* d_taps, int32_t B, int32_t d_v, const void* w_hml, const void* ln_gamma,
                     const void* ln_beta, float ln_eps, int32_t d_g, const void* w_s, int32_t n_bias, float* d_g_out,
                     float* d_bias, void* d_workspace, size_t workspace_bytes, void* stream) {
  sd2_ctx* c = nullptr;
  if (!d_taps || !aligned16(w_hml) || !ln_gamma || !ln_beta || !aligned16(w_s) || !d_g_out || !d_bias || !d_workspace)
    return fail(nullptr, SD2_EINVAL, "null or unaligned argument");
  if (B < 1 || d_v < 1 || d_v % 8 || d_g < 1 || d_g % 8 || n_bias < 1)
    return fail(nullptr, SD2_EINVAL, "need B >= 1 and d_v, d_g multiples of 8");
  if (workspace_bytes < sd2_steer_workspace_bytes(B, d_v, d_g)) return fail(nullptr, SD2_EINVAL, "workspace too small");
  if (reinterpret_cast<uintptr_t>(d_workspace) & 255) return fail(nullptr, SD2_EINVAL, "workspace not 256-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(d_workspace);
  const size_t b = static_cast<size_t>(B);
  void* x_bf = ws;
  float* g_pre = reinterpret_cast<float*>(ws + (b * 3 * d_v * 2 + 255) / 256 * 256);
  void* g_bf = ws + (b * 3 * d_v * 2 + 255) / 256 * 256 + (b * d_g * 4 + 255) / 256 * 256;
  unsigned* err = reinterpret_cast<unsigned*>(static_cast<char*>(g_bf) + (b * d_g * 2 + 255) / 256 * 256);
  CK(cudaMemsetAsync(err, 0, sizeof(unsigned), st));   // the tensor-core GEMMs' wait flag
  CK(gather_rows_bf16(d_taps, 3 * d_v, nullptr, 3 * d_v, B, x_bf, st));
  GemmArgs g{};
  g.x = x_bf; g.ldx = 3 * d_v; g.M = B; g.K = 3 * d_v; g.err = err;
  g.seg[0] = {w_hml, d_g}; g.nseg = 1; g.epi = EPI_STORE; g.out = g_pre; g.ldo = d_g;
  CK(gemm(g, st));
  CK(layernorm(g_pre, ln_gamma, ln_beta, ln_eps, B, d_g, d_g_out, g_bf, st));
  GemmArgs gs{};
  gs.x = g_bf; gs.ldx = d_g; gs.M = B; gs.K = d_g; gs.err = err;
  gs.seg[0] = {w_s, n_bias}; gs.nseg = 1; gs.epi = EPI_STORE; gs.out = d_bias; gs.ldo = n_bias;
  CK(gemm(gs, st));
  return SD2_OK;
}

sd2_status sd2_gemm(const void* d_x, int32_t ldx, int32_t M, int32_t K, const void* d_w, const void* d_w_up,
                    int32_t N, int32_t epilogue, float* d_out, int32_t ldo, void* d_h, const float* d_bias,
                    const int32_t* d_seq, int32_t ld_bias, int32_t impl, void* stream) {
  sd2_ctx* c = nullptr;
  if (!d_x || !d_w || M < 1 || K < 8 || K % 8 || ldx < K || ldx % 8 || N < 1)
    return fail(nullptr, SD2_EINVAL, "bad GEMM shape or null input");
  if (epilogue < EPI_STORE || epilogue > EPI_SILU || epilogue == EPI_QKV)
    return fail(nullptr, SD2_EINVAL, "unknown epilogue");
  if (epilogue == EPI_SWIGLU ? (!d_w_up || !d_h) : epilogue == EPI_SILU ? !d_h : (!d_out || ldo < N))
    return fail(nullptr, SD2_EINVAL, "missing output for the epilogue");
  if (impl < 0 || impl > 2) return fail(nullptr, SD2_EINVAL, "impl must be 0, 1 or 2");
  GemmArgs g{};
  g.x = d_x; g.ldx = ldx; g.M = M; g.K = K;
  g.seg[0] = {d_w, N};
  g.nseg = 1;
  if (epilogue == EPI_SWIGLU) { g.seg[1] = {d_w_up, N}; g.nseg = 2; }
  g.epi = epilogue; g.out = d_out; g.ldo = ldo; g.out_bf = d_h; g.ldh = N;
  g.bias = d_bias; g.ld_bias = ld_bias; g.row_seq = d_seq;
  g.impl = impl == 1 ? 1 : 0;
  // timeout flag of context-free tensor-core launches, allocated once per process (thread-safe)
  static unsigned* const err_word = [] {
    unsigned* w = nullptr;
    if (cudaMalloc(&w, sizeof(unsigned)) != cudaSuccess) return static_cast<unsigned*>(nullptr);
    if (cudaMemset(w, 0, sizeof(unsigned)) != cudaSuccess) {
      cudaFree(w);
      return static_cast<unsigned*>(nullptr);
    }
    return w;
  }();
  if (!err_word) return fail(nullptr, SD2_ENOMEM, "could not allocate the GEMM wait flag");
  g.err = err_word;
  if (impl == 2 && !gemm_tc_supported(g))
    return fail(nullptr, SD2_EINVAL, "shape not supported by the tensor-core GEMM (K % 64, rows % 128)");
  CK(gemm(g, static_cast<cudaStream_t>(stream)));
  return SD2_OK;
}

sd2_status sd2_attention(const float* d_q, int32_t M, int32_t H, int32_t Hkv, int32_t hd, const void* d_pool,
                         int32_t n_blocks, const int32_t* d_table, int32_t bt_stride, int32_t layer,
                         const int32_t* d_row_pos, const int32_t* d_grp_row0, const int32_t* d_grp_nrows,
                         const int32_t* d_grp_seq, int32_t n_groups, int32_t max_rows, int32_t n_splits, int32_t chunk,
                         const int32_t* d_pre_len, int32_t pre_stable, int32_t pre_fresh, void* d_out,
                         uint32_t* d_err, void* stream) {
  sd2_ctx* c = nullptr;
  if (!d_q || !d_pool || !d_table || !d_row_pos || !d_grp_row0 || !d_grp_nrows || !d_grp_seq || !d_out)
    return fail(nullptr, SD2_EINVAL, "null input or output");
  if (M < 1 || n_groups < 0 || Hkv < 1 || H < Hkv || H % Hkv || (hd != 64 && hd != 128) || n_blocks < 1 ||
      bt_stride < 1 || layer < 0 || max_rows < 1 || max_rows * (H / Hkv) > 64)
    return fail(nullptr, SD2_EINVAL, "bad attention shape (hd 64 or 128, max_rows x H/Hkv <= 64)");
  if (n_splits < 1 || n_splits > attention_max_splits() || chunk < 64 || chunk % 64)
    return fail(nullptr, SD2_EINVAL, "n_splits must be 1..attention_max_splits() and chunk a multiple of 64");
  if (d_pre_len && (pre_fresh < 0)) return fail(nullptr, SD2_EINVAL, "pre_fresh must be >= 0");
  AttnArgs at{};
  at.q = d_q;
  at.kv.pool = const_cast<void*>(d_pool); at.kv.table = d_table; at.kv.bt_stride = bt_stride;
  at.kv.n_blocks = n_blocks; at.kv.Hkv = Hkv; at.kv.hd = hd;
  at.layer = layer; at.row_pos = d_row_pos;
  at.grp_row0 = d_grp_row0; at.grp_nrows = d_grp_nrows; at.grp_seq = d_grp_seq; at.n_groups = n_groups;
  at.M = M; at.H = H; at.hd = hd; at.n_splits = n_splits; at.chunk = chunk; at.max_rows = max_rows; at.out = d_out;
  at.pre_len = d_pre_len; at.pre_stable = pre_stable; at.pre_fresh = pre_fresh; at.err = d_err;
  CK(attention(at, static_cast<cudaStream_t>(stream)));
  return SD2_OK;
}

// flat-mode workspace: partial accumulators [Hkv][slots][64][hd] f32, (max, sum) [Hkv][slots][64]
// float2, counters [64][Hkv]
size_t sd2_attention_flat_workspace_bytes(int32_t Hkv, int32_t slots, int32_t hd) {
  if (Hkv < 1 || slots < 1 || hd < 1) return 0;
  const size_t n = static_cast<size_t>(Hkv) * slots * 64;
  return n * hd * 4 + n * 8 + static_cast<size_t>(64) * Hkv * 4;
}

sd2_status sd2_attention_flat(const float* d_q, int32_t M, int32_t H, int32_t Hkv, int32_t hd, const void* d_pool,
                              int32_t n_blocks, const int32_t* d_table, int32_t bt_stride, int32_t layer,
                              const int32_t* d_row_pos, const int32_t* d_grp_row0, const int32_t* d_grp_nrows,
                              const int32_t* d_grp_seq, int32_t n_groups, int32_t max_rows, int32_t slots,
                              int32_t max_ctx, const int32_t* d_pre_len, int32_t pre_stable, int32_t pre_fresh,
                              void* d_work, void* d_out, uint32_t* d_err, void* stream) {
  sd2_ctx* c = nullptr;
  if (!d_q || !d_pool || !d_table || !d_row_pos || !d_grp_row0 || !d_grp_nrows || !d_grp_seq || !d_out ||
      !d_pre_len || !d_work)
    return fail(nullptr, SD2_EINVAL, "null input, output, pre-step lengths or workspace");
  if (reinterpret_cast<uintptr_t>(d_work) % 16) return fail(nullptr, SD2_EINVAL, "workspace must be 16-byte aligned");
  if (M < 1 || Hkv < 1 || H < Hkv || H % Hkv || (hd != 64 && hd != 128) || n_blocks < 1 || bt_stride < 1 ||
      layer < 0 || max_rows < 1 || max_rows * (H / Hkv) > 64)
    return fail(nullptr, SD2_EINVAL, "bad attention shape (hd 64 or 128, max_rows x H/Hkv <= 64)");
  if (n_groups < 1 || n_groups > 64 || slots < n_groups || max_ctx <= 64 || pre_fresh < 0)
    return fail(nullptr, SD2_EINVAL, "flat mode needs 1 <= n_groups <= 64, n_groups <= slots, max_ctx > 64");
  AttnArgs at{};
  at.q = d_q;
  at.kv.pool = const_cast<void*>(d_pool); at.kv.table = d_table; at.kv.bt_stride = bt_stride;
  at.kv.n_blocks = n_blocks; at.kv.Hkv = Hkv; at.kv.hd = hd;
  at.layer = layer; at.row_pos = d_row_pos;
  at.grp_row0 = d_grp_row0; at.grp_nrows = d_grp_nrows; at.grp_seq = d_grp_seq; at.n_groups = n_groups;
  at.M = M; at.H = H; at.hd = hd; at.n_splits = 1; at.chunk = 64 * ((max_ctx + 63) / 64); at.max_rows = max_rows;
  at.out = d_out;
  at.pre_len = d_pre_len; at.pre_stable = pre_stable; at.pre_fresh = pre_fresh; at.err = d_err;
  const size_t n = static_cast<size_t>(Hkv) * slots * 64;
  unsigned char* w = static_cast<unsigned char*>(d_work);
  at.flat = slots;
  at.flat_acc = w;
  at.flat_ml = w + n * hd * 4;
  at.flat_cnt = reinterpret_cast<unsigned*>(w + n * hd * 4 + n * 8);
  CK(attention(at, static_cast<cudaStream_t>(stream)));
  return SD2_OK;
}

sd2_status sd2_swiglu_steered(const float* d_gate, const float* d_up, const float* d_bias, const int32_t* d_seq,
                              int32_t M, int32_t F, void* d_h, void* stream) {
  sd2_ctx* c = nullptr;
  if (!d_gate || !d_up || !d_h || M < 0 || F < 1) return fail(nullptr, SD2_EINVAL, "bad argument");
  CK(swiglu(d_gate, d_up, d_bias, d_seq, M, F, d_h, static_cast<cudaStream_t>(stream)));
  return SD2_OK;
}

}  // extern "C"
