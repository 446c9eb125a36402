/*
 * sd2.h — C ABI of the SD^2 (steered speculative decoding) hot path on one GB300 (sm_103a).
 *
 * One draft-and-verify iteration (Sec. 3 of "Steering Pretrained Drafters during Speculative
 * Decoding", arXiv 2511.09844):
 *   a1  steering vector g_t = LN(W_hml [h_t, m_t, l_t]) from the verifier's hidden states at the
 *       last returned token (Sec. 3.1; layer norm and layers 3, L/2, L-2 from App. A.2), and the
 *       per-layer biases W_s g_t, computed once per drafting stage (Sec. 3.2);
 *   a2  k autoregressive drafter steps whose SwiGLU MLPs are steered as in Eq. 2;
 *   a3  the verifier's parallel forward over the k+1 block positions (Sec. 3.1), which also
 *       writes the hidden states that a1 reads next;
 *   a4  speculative acceptance (greedy, or min(1, p/q) with residual resampling and a bonus
 *       token; Sec. 3.1 and Sec. 4 "Metrics"), then KV-cache rollback of rejected positions.
 *
 * Conventions for every call:
 *   - All pointers prefixed d_ are DEVICE pointers owned by the caller; h_ pointers are host
 *     memory. Weight pointers are borrowed for the lifetime of the context and never written.
 *   - The context owns its own device memory (KV pools, activations, scratch), allocated in
 *     sd2_init and released in sd2_free.
 *   - Work is enqueued on the stream given to sd2_init (a cudaStream_t passed as void*); calls
 *     return without waiting for the GPU, except where stated.
 *   - A call returns SD2_OK or an error code; sd2_last_error(ctx) gives a message. Errors the
 *     GPU detects (non-finite probabilities, a timed-out wait) are latched in a device error word
 *     that sd2_check() reads. No kernel traps or asserts.
 *   - Tensors are row-major. bf16 is IEEE bfloat16 (uint16 bit pattern); f32 is IEEE float.
 */
#ifndef SD2_H
#define SD2_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SD2_OK = 0,
  SD2_EINVAL = 1,     /* bad argument or configuration */
  SD2_ENOMEM = 2,     /* device allocation failed */
  SD2_ECUDA = 3,      /* a CUDA runtime call failed */
  SD2_ECAPACITY = 4,  /* batch, context or prompt exceeds what sd2_init sized */
  SD2_ESTATE = 5,     /* call out of order: init -> prefill -> (step -> accept)* -> free */
  SD2_ENUMERIC = 6,   /* the GPU saw a non-finite logit/probability (latched, see sd2_check) */
  SD2_ETIMEOUT = 7    /* a bounded device-side wait gave up (latched, see sd2_check) */
} sd2_status;

enum { SD2_DTYPE_F32 = 0, SD2_DTYPE_BF16 = 1 };

/* Tensor slots of one decoder layer, in this order, each a bf16 device pointer:
 *   ATTN_NORM [d]            RMSNorm gain before attention
 *   Q [H*hd, d], K [Hkv*hd, d], V [Hkv*hd, d], O [d, H*hd]   (nn.Linear layout: [out, in])
 *   MLP_NORM [d]             RMSNorm gain before the MLP
 *   GATE [F, d], UP [F, d], DOWN [d, F]                        (SwiGLU, Eq. 1 / Eq. 2)     */
enum {
  SD2_W_ATTN_NORM = 0, SD2_W_Q, SD2_W_K, SD2_W_V, SD2_W_O,
  SD2_W_MLP_NORM, SD2_W_GATE, SD2_W_UP, SD2_W_DOWN, SD2_LAYER_SLOTS
};

/* One Llama-style pre-norm decoder (no projection biases, untied lm_head, rotate-half rotary
 * embedding with frequencies rope_theta^(-2i/head_dim)). head_dim must be 64 or 128. */
typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ffn, vocab;
  float rope_theta, norm_eps;
} sd2_lm_config;

typedef struct {
  sd2_lm_config verifier, drafter;   /* same vocab (the paper's pairs share a tokenizer) */
  int32_t d_steer;                   /* width d_g of the steering vector */
  int32_t tap_layers[3];             /* 1-based verifier layers (h, m, l); App. A.2: L-2, L/2, 3 */
  float steer_ln_eps;                /* epsilon of the steering layer norm (App. A.2) */
  int32_t k;                         /* draft length (1..16) */
  int32_t max_batch;                 /* sequences per batch (1..256) */
  int32_t max_ctx;                   /* per-sequence token capacity (prompt + generated + k + 2) */
  int32_t max_prefill_tokens;        /* most prompt tokens one sd2_prefill may carry in total */
  int32_t kv_block;                  /* paged KV-cache block size in tokens; must be 16 */
  int32_t no_steering;               /* 0: SD^2 (Eq. 2 biases in every drafter MLP). 1: the pretrained
                                        drafter alone, the baseline the paper compares with: no steering
                                        stage and no bias (the steering weights may then be null) */
  int32_t steering_site;             /* 0: Eq. 2, the bias added to W_u a before the gating (SD^2);
                                        W_s is [L_D * F_D, d_g]. 1: the "Inv. Bias after MLP" ablation
                                        of Sec. 5, the bias added to each drafter layer's output;
                                        W_s is [L_D * d_D, d_g]. 2: its "Cond. Bias in MLP" ablation,
                                        a per-position bias from a 2-layer MLP of the layer input and
                                        g, used as in Eq. 2 (weights w_c1x, w_c1g, w_c2) */
} sd2_config;

typedef struct {
  const void* embed;                 /* [vocab, d] bf16 */
  const void* final_norm;            /* [d] bf16 */
  const void* lm_head;               /* [vocab, d] bf16 */
  const void* const* layers;         /* HOST array of n_layers*SD2_LAYER_SLOTS device pointers,
                                        layer-major, slot order above; copied by sd2_init */
} sd2_lm_weights;

typedef struct {
  sd2_lm_weights verifier, drafter;
  const void* w_hml;                 /* [d_g, 3*d_v] bf16, columns ordered [h | m | l] (Sec. 3.1) */
  const void* steer_ln_gamma;        /* [d_g] bf16 layer-norm gain (App. A.2) */
  const void* steer_ln_beta;         /* [d_g] bf16 layer-norm shift */
  const void* w_s;                   /* [L_D*F_D, d_g] bf16: rows l*F_D.. give W_s^(l) of Eq. 2
                                        ([L_D*d_D, d_g] with steering_site 1; unused with 2) */
  /* steering_site 2 only: the conditional bias MLP of every drafter layer l,
   * b = W_c2^(l) SiLU(W_c1x^(l) f^(l-1) + W_c1g^(l) g), hidden width d_g (null otherwise) */
  const void* w_c1x;                 /* [L_D*d_g, d_D] bf16 */
  const void* w_c1g;                 /* [L_D*d_g, d_g] bf16 */
  const void* w_c2;                  /* [L_D*F_D, d_g] bf16 */
} sd2_weights;

typedef struct sd2_ctx sd2_ctx;

/* Validate cfg, borrow the weights, allocate the context's device memory and enqueue its
 * initialisation on `stream` (a cudaStream_t). *out receives the context.
 * Errors: SD2_EINVAL (shape unsupported, null pointer), SD2_ENOMEM, SD2_ECUDA. */
sd2_status sd2_init(const sd2_config* cfg, const sd2_weights* w, void* stream, sd2_ctx** out);

/* Start `batch` sequences from their prompts (Sec. 3.1 prefill). d_tokens holds the prompts
 * back to back (int32 ids); h_cu_lens[batch+1] are host prefix offsets into it. h_temperature
 * [batch] per sequence: 0 = greedy (T=0), else sampling at T (applied to both models).
 * The verifier reads each prompt and its last row gives the first new token, written to
 * d_first_token[batch]; the steering vector is read at that row; the drafter reads the prompt
 * under its biases. seed keys the Philox stream of every later random draw.
 * Errors: SD2_EINVAL, SD2_ECAPACITY (batch, prompt length or total tokens too large). */
sd2_status sd2_prefill(sd2_ctx* ctx, int32_t batch, const int32_t* d_tokens, const int32_t* h_cu_lens,
                       const float* h_temperature, uint64_t seed, int32_t* d_first_token);

/* a1 + a2 + a3 of one iteration for every live sequence: compute the steering biases, draft k
 * tokens, and run the verifier over the k+1 block positions. Asynchronous on the ctx stream.
 * Errors: SD2_ESTATE (no prefill, or the previous step was not accepted). */
sd2_status sd2_step(sd2_ctx* ctx);

/* a4: acceptance and rollback for the block of the last sd2_step. Writes, per sequence b,
 * d_tokens[b*(k+1) + t] for t < d_n_emitted[b] (the j kept drafts then one verifier token) and
 * d_n_emitted[b] = j+1 (0 once a sequence has stopped because its capacity is reached).
 * Errors: SD2_ESTATE (no step to accept). */
sd2_status sd2_accept(sd2_ctx* ctx, int32_t* d_tokens, int32_t* d_n_emitted);

/* One whole generation request on host buffers (the serving loop built from the calls above):
 * copies the prompts h_tokens (back to back, h_cu_lens[batch+1] host prefix offsets) to the device,
 * runs sd2_prefill (h_temperature, seed as there) and then sd2_step + sd2_accept until every
 * sequence has max_new tokens or has stopped at the context's capacity, copying each step's
 * emitted tokens back to host memory and waiting for them. Writes h_out[b * max_new + t] for
 * t < h_n_out[b] (the first token from the prefill, then the emitted blocks, cut at max_new).
 * Blocks the calling thread until done. Errors: those of sd2_prefill, sd2_step and sd2_accept. */
sd2_status sd2_generate(sd2_ctx* ctx, int32_t batch, const int32_t* h_tokens, const int32_t* h_cu_lens,
                        const float* h_temperature, uint64_t seed, int32_t max_new, int32_t* h_out,
                        int32_t* h_n_out);

/* Wait for the context's stream and report the device error word (SD2_OK, SD2_ENUMERIC,
 * SD2_ETIMEOUT, or SD2_ECAPACITY when an attention row of a step lay beyond the cache positions
 * that step was planned to write), clearing it. */
sd2_status sd2_check(sd2_ctx* ctx);

/* Release everything the context owns (waits for its stream first). Null is allowed. */
sd2_status sd2_free(sd2_ctx* ctx);

/* Message of the last error on this context (or of the last failed context-free call if ctx
 * is null). Valid until the next call on the same context. */
const char* sd2_last_error(const sd2_ctx* ctx);

/* Use CUDA graphs for sd2_step/sd2_accept (default on). Graphs are captured on first use after
 * each prefill; 0 launches every kernel directly. */
sd2_status sd2_set_graphs(sd2_ctx* ctx, int32_t enable);

/* Read-only views of the context's device buffers, for tests and measurement. `which`:
 *   0 target logits  [B, k+1, V] f32     1 draft logits [B, k, V] f32     2 drafts x^ [B, k] i32
 *   3 verifier taps  [B, k+1, 3, d_v] f32 (order h, m, l)   4 steering vector g [B, d_g] f32
 *   5 steering biases [B, L_D*F_D] f32 ([B, L_D*d_D] with steering_site 1)   6 committed tokens [B, max_ctx] i32
 *   7 per-sequence state [B, 4] i32: committed length n, drafter cached length, j, stopped
 *   8 iteration counter [1] i32 (the `step` of the Philox counters; 0 = prefill)
 * *d_ptr, *n_elems and *dtype (SD2_DTYPE_*) describe the buffer; B is the prefilled batch. */
sd2_status sd2_debug_buffer(const sd2_ctx* ctx, int32_t which, void** d_ptr, int64_t* n_elems,
                            int32_t* dtype);

/* Per-kernel-class timing of the iterations that follow, measured with CUDA events on the ctx
 * stream (graphs are not used while profiling is on). sd2_profile_read returns, per class,
 * launches, total milliseconds and algorithmic bytes. Classes: 0 GEMM (weight streaming),
 * 1 attention, 2 acceptance, 3 sampling, 4 other, 5 verify stage (a3), 6 draft stage (a2),
 * 7 steering stage (a1). */
sd2_status sd2_profile(sd2_ctx* ctx, int32_t enable);
sd2_status sd2_profile_read(sd2_ctx* ctx, int64_t* launches, double* ms, double* bytes, int32_t n_classes);

/* Stage timing inside the captured step: with it enabled, every following sd2_step records CUDA
 * events (external event nodes in the graph) before the steering stage (a1), between the k
 * drafter steps (a2) and around the verifier forward (a3); the kernels between them run exactly
 * as in an untimed step. Toggling re-captures the step graph. sd2_stage_read waits for the ctx
 * stream and writes the last step's milliseconds: ms[0] steering, ms[1] all k drafter steps,
 * ms[2] verifier forward. SD2_ESTATE when no timed step has run. */
sd2_status sd2_stage_timing(sd2_ctx* ctx, int32_t enable);
sd2_status sd2_stage_read(sd2_ctx* ctx, double* ms);

/* Failure-detection hooks for tests (the paper has no counterpart).
 * sd2_debug_fail_alloc(after): process-wide; the device allocation of a context (sd2_init) that
 * comes `after` allocations from now fails as if cudaMalloc had, once: the call that makes it
 * returns SD2_ENOMEM and releases what it had allocated. A negative value disarms the hook.
 * sd2_debug_expire_wait(ctx, cycles): enqueue on the context's stream one bounded device wait of
 * the kind every kernel wait is (an mbarrier wait with a clock budget), on a barrier nothing
 * arrives on, with a budget of `cycles` (1 .. the kernels' own budget of about 2 s): it gives up,
 * latches the time-out in the context's error word and returns, so the next sd2_check reports
 * SD2_ETIMEOUT and the context stays usable. */
sd2_status sd2_debug_fail_alloc(int32_t after);
sd2_status sd2_debug_expire_wait(sd2_ctx* ctx, int64_t cycles);

/* In-graph timing of the weight-streaming GEMM: with it enabled, every following sd2_step (graph
 * replayed as usual, re-captured when this is toggled) has each tensor-core GEMM launch record
 * three %globaltimer stamps (ns) into a slot of its own: the earliest entry of any of its CTAs,
 * the earliest return from the programmatic wait (the kernel before it has completed) and the
 * latest CTA exit. The launches are otherwise exactly those of an untimed step.
 * sd2_gemm_timing_read waits for the ctx stream and gives, for the last timed step, *n launches
 * in stream order and, for the first min(*n, cap): stamps[3 i .. 3 i + 2], the launch's
 * algorithmic bytes (weights + activations in + outputs) and its stage (0 steering, 1..k drafter
 * step i, k + 1 verify). SD2_ESTATE when no timed step has run. */
sd2_status sd2_gemm_timing(sd2_ctx* ctx, int32_t enable);
sd2_status sd2_gemm_timing_read(sd2_ctx* ctx, int32_t cap, int32_t* n, uint64_t* stamps, double* bytes,
                                int32_t* stage);

/* ---------------------------------------------------------------------------------------------
 * Standalone kernels (no context): the acceptance and steering steps on caller buffers.
 * ------------------------------------------------------------------------------------------- */

/* Scratch bytes sd2_accept_logits needs for batch B and draft length k. */
size_t sd2_accept_workspace_bytes(int32_t B, int32_t k);

/* Speculative acceptance of B independent blocks (a4 without rollback), Sec. 3.1:
 *   d_target [B, k+1, V], d_draft [B, k, V] logits of `dtype` (SD2_DTYPE_F32 or _BF16);
 *   row i of d_target is the verifier's distribution after block input i, row i-1 of d_draft
 *   is the distribution q_i draft i was drawn from; d_xhat [B, k] int32 drafts;
 *   d_temperature [B] f32 (0 = greedy). Random draws use Philox4x32-10 (Salmon et al. SC'11)
 *   with key (seed mod 2^32, seed >> 32) and counter (c0, purpose<<16 | i, b, step):
 *   the uniform of draft i's test is word 0 of (0, 1<<16 | i, b, step); the replacement or
 *   bonus token drawn from block row i uses, for vocabulary entry v, word v&3 of
 *   (v>>2, 2<<16 | i, b, step); u = (2*(word>>9)+1) * 2^-24. Outputs d_tokens [B, k+1] int32
 *   (first d_n[b] entries valid) and d_n [B] = accepted + 1.
 *   d_workspace: caller device scratch of sd2_accept_workspace_bytes(B, k) bytes, 256-byte
 *   aligned; contents need not be initialised. Errors: SD2_EINVAL (sizes, null, alignment). */
sd2_status sd2_accept_logits(const void* d_target, const void* d_draft, int32_t dtype,
                             const int32_t* d_xhat, const float* d_temperature, int32_t B, int32_t k,
                             int32_t V, uint64_t seed, uint32_t step, int32_t* d_tokens, int32_t* d_n,
                             void* d_workspace, size_t workspace_bytes, void* stream);

/* Steering step a1 on caller buffers: g = LN(W_hml [h; m; l]) * gamma + beta and biases
 * W_s g for B sequences (Sec. 3.1, Eq. 2, App. A.2).
 *   d_taps [B, 3, d_v] f32 in the order (h, m, l); weights bf16 as in sd2_weights;
 *   outputs d_g [B, d_g] f32 and d_bias [B, n_bias] f32, n_bias = L_D * F_D.
 *   Both projections run on the tensor-core GEMM where the shapes allow it (d_g and n_bias
 *   multiples of 128, 3 d_v and d_g multiples of 64), else on CUDA cores.
 *   d_workspace: device scratch of sd2_steer_workspace_bytes(B, d_v, d_g) bytes, 256-byte aligned;
 *   contents need not be initialised (it also holds the GEMM's wait flag, reset by each call), so
 *   calls whose GPU work overlaps must not share it. Errors: SD2_EINVAL (null, unaligned, sizes,
 *   workspace too small), SD2_ECUDA. No device memory is allocated. */
size_t sd2_steer_workspace_bytes(int32_t B, int32_t d_v, int32_t d_g);
sd2_status sd2_steer(const float* d_taps, int32_t B, int32_t d_v, const void* w_hml, const void* ln_gamma,
                     const void* ln_beta, float ln_eps, int32_t d_g, const void* w_s, int32_t n_bias,
                     float* d_g_out, float* d_bias, void* d_workspace, size_t workspace_bytes, void* stream);

/* Weight-streaming GEMM of the decoder on caller buffers, Y[m, n] = sum_k X[m, k] W[n, k]:
 *   d_x [M, ldx] bf16 (first K columns used), d_w [N, K] bf16 (nn.Linear layout).
 *   epilogue 0: d_out[m*ldo + n] = Y (f32); 1: d_out[m*ldo + n] += Y (the residual add), plus
 *      d_bias[seq[m]*ld_bias + n] when d_bias is given (the after-MLP steering site);
 *   2: the steered SwiGLU of Eq. 2 with d_w = W_gate, d_w_up = W_up (both [N, K]):
 *      d_h[m*N + f] = bf16((up + d_bias[seq[m]*ld_bias + f]) * SiLU(gate)), d_bias/d_seq optional;
 *   4: d_h[m*N + n] = bf16(SiLU(Y + d_bias[seq[m]*ld_bias + n])), d_bias/d_seq optional (the hidden
 *      layer of the conditional bias MLP).
 *   impl 0: tensor cores (tcgen05, TMA) where the shape allows (K % 64 == 0; N % 128 == 0, or
 *   N % 64 == 0 for epilogue 2), else CUDA cores; 1: CUDA cores; 2: tensor cores or SD2_EINVAL.
 *   No device memory is allocated except, once, a 4-byte error word. */
sd2_status sd2_gemm(const void* d_x, int32_t ldx, int32_t M, int32_t K, const void* d_w, const void* d_w_up,
                    int32_t N, int32_t epilogue, float* d_out, int32_t ldo, void* d_h, const float* d_bias,
                    const int32_t* d_seq, int32_t ld_bias, int32_t impl, void* stream);

/* Causal grouped-query attention of the decoder layers (Sec. 3.2, the SwiGLU decoders of drafter and
 * verifier) over a paged KV cache, on caller buffers (the kernel of the engine's steps).
 *   d_q [M, H, hd] f32: rotated queries of M rows; hd 64 or 128; H a multiple of Hkv.
 *   d_pool bf16 [L][n_blocks][2 (K, V)][Hkv][16][hd]; d_table int32 [n_seq, bt_stride]: the block
 *   holding positions 16 i .. 16 i + 15 of sequence s (ids in [0, n_blocks)); `layer` selects L.
 *   Groups g < n_groups: rows d_grp_row0[g] .. d_grp_row0[g] + d_grp_nrows[g] - 1 belong to sequence
 *   d_grp_seq[g]; row m (position d_row_pos[m]) attends to its sequence's positions 0 .. d_row_pos[m].
 *   max_rows >= every d_grp_nrows, max_rows * H / Hkv <= 64. The context is cut into n_splits chunks
 *   of `chunk` positions (a multiple of 64; 1 <= n_splits <= 16 where the device schedules clusters
 *   of 16 CTAs, else 8); positions at or beyond n_splits * chunk or 16 * bt_stride are not read.
 *   d_pre_len (may be null): per sequence, positions below d_pre_len[s] + pre_stable are read before
 *   the programmatic wait (they must not be written by the kernel launched just before on the
 *   stream), and every row lies below d_pre_len[s] + pre_stable + pre_fresh; cache rows between
 *   the two bounds must hold finite values.
 *   d_out [M, H * hd] bf16. d_err (may be null): a device word or-ed with 2 (a merge wait timed out)
 *   or 4 (a row lay beyond the d_pre_len bound). No device memory is allocated. */
sd2_status sd2_attention(const float* d_q, int32_t M, int32_t H, int32_t Hkv, int32_t hd, const void* d_pool,
                         int32_t n_blocks, const int32_t* d_table, int32_t bt_stride, int32_t layer,
                         const int32_t* d_row_pos, const int32_t* d_grp_row0, const int32_t* d_grp_nrows,
                         const int32_t* d_grp_seq, int32_t n_groups, int32_t max_rows, int32_t n_splits, int32_t chunk,
                         const int32_t* d_pre_len, int32_t pre_stable, int32_t pre_fresh, void* d_out,
                         uint32_t* d_err, void* stream);

/* Bytes of device workspace sd2_attention_flat needs for `slots` CTAs per KV head. */
size_t sd2_attention_flat_workspace_bytes(int32_t Hkv, int32_t slots, int32_t hd);

/* The same attention laid out as the engine runs decode steps over many sequences of ragged lengths
 * (flat mode): `slots` CTAs per KV head are shared out over the groups on the device, each group
 * taking ceil(t_g / t) of them (t_g its visible length d_pre_len[s] + pre_stable + pre_fresh in tiles
 * of 64 positions, t the smallest tile count per CTA for which all groups fit, at most 32 CTAs a
 * group); the splits of a group merge through the workspace and the group's last split writes its
 * output. Same arguments as sd2_attention except: d_pre_len is required; 1 <= n_groups <= 64 and
 * n_groups <= slots; max_ctx (> 64) bounds every visible length; d_work is
 * sd2_attention_flat_workspace_bytes(Hkv, slots, hd) bytes of device memory, 16-byte aligned, zeroed
 * by the caller before its first use and left zeroed by every call that completes (its counters reset
 * themselves), used by one call at a time. Errors: SD2_EINVAL for a bad shape or a null pointer; the
 * d_err bits as in sd2_attention. No device memory is allocated. */
sd2_status sd2_attention_flat(const float* d_q, int32_t M, int32_t H, int32_t Hkv, int32_t hd, const void* d_pool,
                              int32_t n_blocks, const int32_t* d_table, int32_t bt_stride, int32_t layer,
                              const int32_t* d_row_pos, const int32_t* d_grp_row0, const int32_t* d_grp_nrows,
                              const int32_t* d_grp_seq, int32_t n_groups, int32_t max_rows, int32_t slots,
                              int32_t max_ctx, const int32_t* d_pre_len, int32_t pre_stable, int32_t pre_fresh,
                              void* d_work, void* d_out, uint32_t* d_err, void* stream);

/* Choose the GEMM of a context: 0 tensor cores where the shape allows (default), 1 CUDA cores.
 * Drops captured graphs. */
sd2_status sd2_set_gemm_impl(sd2_ctx* ctx, int32_t impl);

/* Run each drafter step's decoder layers as one persistent cooperative kernel (1, wherever the
 * drafter's shape and the step's rows allow it: at most 16 rows, d_model <= 2048) or as one kernel
 * per projection and attention (0, the default: faster on GB300 at batch 1). Either way the same
 * arithmetic of a2. Only with the tensor-core GEMM (sd2_set_gemm_impl 0). Drops captured graphs. */
sd2_status sd2_set_drafter_chain(sd2_ctx* ctx, int32_t enable);

/* Decode steps of one sequence (batch 1): run each layer's attention inside its O projection
 * (1, where the model allows it: head dim 64, 2..8 KV heads, rows x heads per KV head <= 16,
 * context <= 4096, the projection's tiles x KV heads <= the SM count) or as a kernel of its own
 * (0, the default: faster on GB300, where the fused kernel's shared memory keeps the neighbouring
 * kernels from overlapping it). Either way the same arithmetic. Drops captured graphs. */
sd2_status sd2_set_fused_attention(sd2_ctx* ctx, int32_t enable);

/* Steered SwiGLU activation of Eq. 2 on caller buffers (the injection step of a2):
 *   h[m, f] = (up[m, f] + bias[seq[m], f]) * SiLU(gate[m, f]) as bf16, with gate/up [M, F] f32,
 *   bias [*, F] f32 (row seq[m]; d_seq may be null for bias row 0), h [M, F] bf16. */
sd2_status sd2_swiglu_steered(const float* d_gate, const float* d_up, const float* d_bias,
                              const int32_t* d_seq, int32_t M, int32_t F, void* d_h, void* stream);

/* The acceptance of sd2_accept_logits without any device allocation by the caller or by the
 * library. (An addition of this library: the paper has no counterpart.) It is for callers that
 * cannot call cudaMalloc, for example code living in a process whose device memory is owned by
 * another component's allocator, or a loop that must not risk the device-wide synchronisation a
 * cudaMalloc/cudaFree can cause. Arguments and outputs are those of sd2_accept_logits, minus the
 * workspace: the scratch is a fixed 256 KiB device array inside the library, held on every GPU
 * that loads it until the process exits. Its acceptance tables take 16*B*(2k+1) + 28*B + 64
 * bytes of it and the error word sits in its last 256 bytes, so requests above 261888 bytes of
 * tables return SD2_ECAPACITY (B = 256 with k = 16 needs 142400 bytes; k = 16 allows B <= 470).
 *   - The array's device address belongs to a CUDA context: the first call in each context (the
 *     device's primary context, or one the caller made current) looks it up with
 *     cudaGetSymbolAddress, and later calls in that context reuse it. Make that first call before
 *     any stream capture.
 *   - Every call on a device shares the one array and leaves its contents behind; the call
 *     clears what must start at zero. Calls whose GPU work overlaps (other streams, other host
 *     threads) race on the array: order them on one stream.
 *   - Errors: the status, with the text in sd2_last_error(NULL). Non-finite logits are found on
 *     the GPU after the call has returned: sd2_accept_logits_noalloc_check reports them. */
sd2_status sd2_accept_logits_noalloc(const void* d_target, const void* d_draft, int32_t dtype,
                                     const int32_t* d_xhat, const float* d_temperature, int32_t B,
                                     int32_t k, int32_t V, uint64_t seed, uint32_t step,
                                     int32_t* d_tokens, int32_t* d_n, void* stream);

/* Error word of the last sd2_accept_logits_noalloc call in the current context: waits for
 * `stream` (the stream that call was given), reads the word from the fixed array, clears it and
 * returns SD2_ENUMERIC if that call saw a non-finite logit, else SD2_OK (SD2_ECUDA if a CUDA call
 * fails). Allocates nothing. Each acceptance call clears the word when it starts, so the check
 * reports the last call only. */
sd2_status sd2_accept_logits_noalloc_check(void* stream);

#ifdef __cplusplus
}
#endif
#endif /* SD2_H */
