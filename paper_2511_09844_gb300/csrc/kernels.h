// Host-side launchers of the SD^2 kernels (one declaration per kernel family). Every
// launcher enqueues on `st` and returns the launch's cudaError_t.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <utility>

namespace sd2 {

// Launch with programmatic stream serialisation (see pdl_wait / pdl_trigger in common.cuh).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// The same with a 1-D thread-block cluster of `cluster` CTAs (1 = no cluster).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                               int cluster, Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  int n = 1;
  if (cluster > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = static_cast<unsigned>(cluster);
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    n = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------- weight-streaming GEMM
// Y[m, n] = sum_k X[m, k] W[n, k] for m < M, with W the row concatenation of up to three
// bf16 segments (e.g. W_q | W_k | W_v). X is bf16 with row stride ldx; K % 8 == 0.
enum GemmEpilogue {
  EPI_STORE = 0,    // out[m*ldo + n] = y (f32)
  EPI_ADD = 1,      // out[m*ldo + n] += y (f32 residual stream)
  EPI_SWIGLU = 2,   // Eq. 2: h[m*ldh + f] = bf16((up + bias[seq[m]*ld_bias + f]) * SiLU(gate));
                    //   segments: seg0 = W_gate [F, K], seg1 = W_up [F, K]
  EPI_QKV = 3,      // segments W_q | W_k | W_v: rotary embedding on q and k, q -> q_out [M, H, hd] f32,
                    //   k and v of valid rows -> the paged KV cache of `layer` at (row_seq, row_pos)
  EPI_SILU = 4,     // out_bf[m*ldh + n] = bf16(SiLU(y + bias[seq[m]*ld_bias + n])) (bias optional)
};
struct GemmSeg {
  const void* w;
  int rows;
};
struct GemmArgs {
  const void* x;
  int ldx, M, K;
  GemmSeg seg[3];
  int nseg;
  int epi;
  float* out;
  int ldo;
  void* out_bf;
  int ldh;
  const float* bias;
  int ld_bias;
  const int* row_seq;
  // the device error word (bounded waits) and the implementation: 0 = tensor cores when the
  // shape allows, 1 = CUDA cores
  unsigned* err;
  int impl;
  // In-graph timing (tensor-core path; may be null): three words per launch, set with atomics on
  // %globaltimer (ns): [0] earliest CTA entry, [1] earliest return from the programmatic wait (the
  // predecessor grid has completed), [2] latest CTA exit. The caller presets [0], [1] to ~0 and
  // [2] to 0.
  unsigned long long* stamp;
  // EPI_QKV
  float* q_out;
  void* kv_pool;
  const int* kv_table;
  int kv_bt_stride, kv_n_blocks, n_heads, n_kv_heads, head_dim, layer;
  const float* rope_cs;
  const int* row_pos;
  const int* row_valid;
  // RMSNorm fused across GEMMs (tensor-core path only). Producer (EPI_ADD with norm_out set):
  // besides x_new = out + y it writes norm_out[m * ldo + n] = bf16(x_new[m, n] * norm_gamma[n]),
  // the sums of squares of x_new over its slices of n, norm_ssq_out[part * ld_ssq + m] for
  // part < gemm_norm_parts(this launch), and x_new into tap slot s (tap_mask bit s) of rows with
  // tap_row[m] >= 0: tap[(tap_row[m] * 3 + s) * ldo + n].
  const void* norm_gamma;
  void* norm_out;
  float* norm_ssq_out;
  float* tap;
  const int* tap_row;
  int tap_mask;
  // Consumer (norm_ssq_in set): each output of token m is scaled by
  // rsqrt(sum_{p < norm_parts} norm_ssq_in[p * ld_ssq + m] / norm_d + norm_eps), the RMSNorm of
  // the producer's x_new, before the epilogue (the GEMM's input being bf16(x_new * gamma)).
  const float* norm_ssq_in;
  int norm_parts, norm_d;
  float norm_eps;
  int ld_ssq;
  // Fused decode attention (tensor-core path, gemm_attn_supported): with attn_q set, the token
  // operand x is not read; it is the causal attention output of the M rows, all of sequence
  // *attn_seq (a plan table written before the step), computed in the kernel from attn_q
  // [M, n_heads, 64] f32 and the paged cache (kv_* fields, layer, row_pos). Cache positions below
  // attn_pre_len[seq] + attn_pre_stable were written before the step; every row lies below that
  // + attn_pre_fresh, and the cache rows up to there hold finite values.
  const float* attn_q;
  const int* attn_seq;
  const int* attn_pre_len;
  int attn_pre_stable, attn_pre_fresh;
};
// Number of sums-of-squares slices a producer launch with these arguments writes.
int gemm_norm_parts(const GemmArgs& a);
// Dispatches to the tcgen05 kernel (gemm_tc.cu) when impl != 1 and gemm_tc_supported holds, else
// to the CUDA-core kernel (gemm_simt.cu).
cudaError_t gemm(const GemmArgs& a, cudaStream_t st);
bool gemm_tc_supported(const GemmArgs& a);
// Whether the fused decode attention (attn_q) can run for these arguments on this device.
bool gemm_attn_supported(const GemmArgs& a);
cudaError_t gemm_tc(const GemmArgs& a, unsigned* err, cudaStream_t st);
int gemm_tc_token_tile(int M);
cudaError_t gemm_simt(const GemmArgs& a, cudaStream_t st);

// 2-D bf16 TMA map (CUtensorMap, 128 bytes) of a row-major [rows, K] weight: boxes of box_rows x 64
// elements with the 128-byte swizzle (gemm_tc.cu).
bool encode_weight_map(void* map, const void* w, int rows, int K, int box_rows);
int sm_count_cached();

// ---------------------------------------------------------------- decoder elementwise
// out[m, :w] = bf16(x[m * ld + 0 .. w-1]) for m < M.
cudaError_t rows_to_bf16(const float* x, int ld, int M, int w, void* out, cudaStream_t st);
// x[m] = embed[tok[m]] (f32), a[m] = bf16(RMSNorm(x[m]) * gamma); ids are clamped to [0, vocab).
cudaError_t embed_rmsnorm(const int* tok, const void* embed, const void* gamma, float eps, int M, int d, int vocab,
                          float* x, void* a, cudaStream_t st);
// Producer form for the fused RMSNorm: x[m] = embed[tok[m]], a[m] = bf16(x[m] * gamma) and
// ssq[m] = sum_n x[m, n]^2 (one slice).
cudaError_t embed_scaled(const int* tok, const void* embed, const void* gamma, int M, int d, int vocab, float* x,
                         void* a, float* ssq, cudaStream_t st);
// a[i] = bf16(RMSNorm(x[src(i)]) * gamma) for i < M, src(i) = rows ? rows[i] : i.
// Taps: for each of up to 3 slots s with tap_mask bit s, tap[(tap_row[src] * 3 + s) * d] = x[src]
// for source rows whose tap_row >= 0 (tap_row may be null = identity).
cudaError_t rmsnorm(const float* x, const int* rows, const void* gamma, float eps, int M, int d, void* a,
                    float* tap, const int* tap_row, int tap_mask, cudaStream_t st);
// Rotary embedding + paged KV append. qkv [M, (H + 2 Hkv) hd] f32 -> q [M, H, hd] f32 (rotated);
// rotated k and v go to the cache of `layer` at each valid row's (seq, pos).
struct KVCache {
  void* pool;          // bf16 [L][n_blocks][2][Hkv][16][hd]
  const int* table;    // [max_batch, bt_stride] block ids
  int bt_stride, n_blocks, Hkv, hd;
};
cudaError_t rope_append(const float* qkv, const float* rope_cs, int M, int H, int Hkv, int hd, const int* row_seq,
                        const int* row_pos, const int* row_valid, const KVCache& kv, int layer, float* q,
                        cudaStream_t st);
// Steering layer norm: g = LN(x) * gamma + beta (f32 and bf16 copies), rows of width d.
cudaError_t layernorm(const float* x, const void* gamma, const void* beta, float eps, int B, int d, float* g,
                      void* g_bf, cudaStream_t st);
// Steered SwiGLU on precomputed projections (standalone form of EPI_SWIGLU).
cudaError_t swiglu(const float* gate, const float* up, const float* bias, const int* seq, int M, int F, void* h,
                   cudaStream_t st);
// f32 -> bf16 rows: out[b, :] = src[b*ld_src + off(b)*width .. +width], off(b) = idx ? idx[b] : 0.
cudaError_t gather_rows_bf16(const float* src, int ld_src, const int* idx, int width, int B, void* out,
                             cudaStream_t st);

// ---------------------------------------------------------------- attention
// Causal paged attention for query rows grouped by sequence: group g covers rows
// grp_row0[g] .. +grp_nrows[g] of sequence grp_seq[g]; row r attends to cache positions
// 0..row_pos[r]. The context is cut into splits of `chunk` positions (a multiple of 64);
// with n_splits == 1 the result goes straight to out, otherwise the last split of each
// (group, KV head) to finish merges the partials.
struct AttnArgs {
  const float* q;        // [M, H, hd] rotated queries
  KVCache kv;
  int layer;
  const int* row_pos;
  const int* grp_row0;
  const int* grp_nrows;
  const int* grp_seq;
  int n_groups, M, H, hd;
  int n_splits, chunk;   // context splits (<= attention_max_splits(), one cluster) of `chunk` positions (a multiple of 64)
  int max_rows;          // upper bound of grp_nrows (max_rows x heads per KV head <= 64)
  void* out;             // [M, H * hd] bf16
  // Decode steps: per sequence, cache positions [0, pre_len[seq] + pre_stable) were written before
  // the step's first kernel (their K/V rows are loaded before the programmatic wait), and the rows
  // of the step lie below pre_len[seq] + pre_stable + pre_fresh; the cache rows in between must
  // hold finite values (the pool starts zeroed). nullptr: every row is loaded after the wait.
  const int* pre_len;
  int pre_stable, pre_fresh;
  unsigned* err;         // ERR_TIMEOUT (split merge), ERR_RANGE (a row outside the planned range); may be null
  // Context clusters: R > 1 clusters of n_splits CTAs each share the context (R * n_splits splits of
  // `chunk`); their partials meet in part_acc / part_ml ([n_groups][Hkv][R][64 * hd/4] float4 /
  // float2) and the last owner of each share, counted in part_cnt ([n_groups][Hkv][n_splits],
  // zero-initialised, self-resetting), writes the output. Needs n_splits >= 2.
  int n_ctx_clusters = 1;
  void* part_acc = nullptr;
  void* part_ml = nullptr;
  void* part_cnt = nullptr;
  // Flat mode (decode steps of several row groups, ragged lengths): `flat` > 0 CTAs ("slots") per KV
  // head, one-CTA clusters, shared out over the groups on the device from their pre-step lengths so
  // that no slot holds more tiles than needed; a group's splits meet in flat_acc ([Hkv][flat][64][hd]
  // f32, unnormalised) and flat_ml ([Hkv][flat][64] float2: max, sum), counted in flat_cnt
  // ([n_groups][Hkv], zero-initialised, self-resetting); the last split of a group writes its output.
  // Needs pre_len, n_splits == 1, n_ctx_clusters == 1, n_groups <= flat and n_groups <= 64.
  int flat = 0;
  void* flat_acc = nullptr;
  void* flat_ml = nullptr;
  unsigned* flat_cnt = nullptr;
};
cudaError_t attention(const AttnArgs& a, cudaStream_t st);
// Most context splits (= CTAs of one cluster) attention takes on this device: 16 where clusters of
// 16 CTAs can be scheduled, else 8.
int attention_max_splits();
// CTAs of one attention launch an SM can hold at once for head dim hd (4 for 64, 2 for 128).
int attention_ctas_per_sm(int hd);
// Clusters of the launch `a` describes (n_splits CTAs each, with the shared memory attention()
// would give them) that the device holds at once: the occupancy calculator's count, which sees how
// clusters pack into the GPCs where the per-SM count above does not. 0 for shapes attention() rejects.
int attention_max_clusters(const AttnArgs& a);

// ---------------------------------------------------------------- persistent layer chain
// Every decoder layer of one forward pass over at most 16 token rows in one cooperative launch
// (chain.cu): the projections stream their weights through one TMA ring across grid-wide
// barriers, split-K partials are summed by the phase that reads them, attention runs between.
struct ChainPlan {                   // one decoder, prepared once
  int L = 0, d = 0, H = 0, Hkv = 0, hd = 0, F = 0;
  float eps = 0.f;
  const void* embed = nullptr;       // bf16 [vocab, d]
  int vocab = 0;
  KVCache kv{};
  const float* rope_cs = nullptr;    // float2 [max_ctx, hd / 2]
  int n_cta = 0, sp_q = 0, sp_o = 0, sp_d = 0, max_splits = 0;
  void* dev = nullptr;               // tensor maps and norm gains of every layer (chain_prepare)
  float *xbuf = nullptr, *pq = nullptr, *po = nullptr, *pd = nullptr, *pa = nullptr;
  void* h = nullptr;
  unsigned* sync = nullptr;
};
// Shape checks and work split of a decoder; false if the chain does not take it.
bool chain_plan(ChainPlan& p, int L, int d, int H, int Hkv, int hd, int F, int vocab, float eps, int max_splits);
// Device bytes chain_prepare needs for p (tables + scratch).
size_t chain_device_bytes(const ChainPlan& p);
// Writes the tables into `block` (chain_device_bytes of 256-aligned device memory) and points the
// scratch into it. w = host array of L * SD2_LAYER_SLOTS device weight pointers.
cudaError_t chain_prepare(ChainPlan& p, const void* const* w, const void* embed, const KVCache& kv,
                          const float* rope_cs, void* block);
struct ChainRun {
  int M = 0;                         // token rows (<= 16)
  const int *tok = nullptr, *row_pos = nullptr, *row_seq = nullptr, *row_valid = nullptr;
  const int *grp_row0 = nullptr, *grp_nrows = nullptr, *grp_seq = nullptr;
  int n_groups = 0, n_splits = 1, chunk = 64, max_rows = 1;
  const float* bias = nullptr;       // steering biases [seq][L * F] (Eq. 2), null for none
  int ld_bias = 0;
  float* x_out = nullptr;            // [M, d] residual stream after the last layer
  unsigned* err = nullptr;
};
bool chain_supported(const ChainPlan& p, const ChainRun& r);
cudaError_t chain_forward(const ChainPlan& p, const ChainRun& r, cudaStream_t st);


// ---------------------------------------------------------------- sampling / acceptance
// Scratch layout used by the acceptance kernels for R = B(2k+1) rows and B sequences.
struct AcceptScratch {
  unsigned long long* rowkey;   // [R] packed (max of z/T or z, argmax)
  unsigned long long* rowsum;   // [R] fixed-point normaliser
  unsigned long long* slot;     // [B, 2] race maxima (residual, log-form)
  int* counter;                 // [B] CTAs finished in the race
  int* jmode;                   // [B, 2] j and mode
};
size_t accept_scratch_bytes(int B, int k);
// Philox key of the sampling kernels: `value`, or the word at `ptr` when ptr is set (so that a
// captured step can take a new request's seed without being captured again).
struct Seed {
  unsigned long long value;
  const unsigned long long* ptr;
};
AcceptScratch accept_scratch_carve(void* base, int B, int k);
// Acceptance of B blocks. logits are f32 (dtype 0) or bf16 (1); target row stride ld_t
// between consecutive rows of one sequence is V and sequence stride (k+1)V, likewise the draft
// with kV. Writes tokens [B, k+1] and n [B]; n_live (optional) masks stopped sequences
// (n_live[b] == 0 -> n[b] = 0). step_ptr (optional) overrides `step` from device memory.
cudaError_t accept_blocks(const void* target, const void* draft, int dtype, const int* xhat, const float* temp,
                          int B, int k, int V, Seed seed, unsigned step, const int* step_ptr,
                          const int* live, int* tokens, int* n, const AcceptScratch& s, unsigned* err,
                          cudaStream_t st);
// Token from one row per sequence (draft sample or bonus/first token): T = 0 -> argmax,
// else the exponential race argmax_v (z_v/T - ln(-ln u_v)) with u from counter
// (v>>2, purpose<<16 | i, b, step). Row of sequence b at logits + b*ld. The result goes to
// out[b*ld_out] and, if out2, out2[b*ld_out2].
cudaError_t sample_rows(const float* logits, long long ld, int B, int V, const float* temp, Seed seed,
                        int purpose, int i, const int* step_ptr, unsigned step, int* out, int ld_out, int* out2,
                        int ld_out2, unsigned long long* slot, int* counter, unsigned* err, cudaStream_t st);

}  // namespace sd2
