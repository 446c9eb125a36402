// Weight-streaming GEMM on the 5th-generation tensor cores: Y[m, n] = sum_k X[m, k] W[n, k] with
// the decoder's fused epilogues (store, residual add, steered SwiGLU of Eq. 2).
//
// The few token rows of a decode or verify step (M <= 256 per tile) cannot fill the M = 128
// side of tcgen05.mma, so the operands are swapped: each tile is 128 weight rows (the MMA's M)
// against NT token rows (the MMA's N, a multiple of 16), accumulating in TMEM. Weights and
// tokens are K-major bf16 tiles of 64 elements (128 bytes) per stage, loaded by TMA with the
// 128-byte swizzle that the UMMA shared-memory descriptors expect.
//
// Work split. A launch has T = (weight tiles) x (token tiles) output tiles of K/64 k-blocks each.
// When T is small (few, tall weight matrices) each tile's K range is split over sp <= 8 CTAs
// that form one thread-block cluster. The tile's rows are kept in pairs (SwiGLU gate/up, rotary
// partners), and each rank owns a share of the pairs: every rank stores its fp32 partial of each
// pair into the owner's shared memory (distributed shared memory), one cluster barrier later the
// owner sums the partials in rank order from its own shared memory and runs the epilogue. No
// partial leaves the SMs, no CTA waits on a remote load, and no CTA waits on global atomics. When T is large, sp = 1 and each CTA streams whole tiles, double-buffering its TMEM
// accumulator across tiles. Either way ~152 CTAs stream at once, and with the stage ring kept
// within half an SM's shared memory a second CTA (the next kernel's, under programmatic
// dependent launch) can start on the same SM and prefetch its weights.
//
// Warp roles (192 threads): warp 0 issues TMA loads into a ring of stages, warp 1 issues the
// MMAs (one thread) and owns the TMEM allocation, warps 2-5 read the TMEM accumulators back
// (each warp its 32-lane quarter) and run the epilogue. Every wait is bounded by a clock budget;
// on expiry the kernel records ERR_TIMEOUT, drains what it issued and returns.
#include <cuda.h>
#include <limits.h>

#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace sd2 {
namespace {

using namespace tc;

constexpr int kWRows = 128;          // weight rows per tile = the MMA's M
constexpr int kBK = 64;              // K per stage (128 bytes of bf16)
constexpr int kThreads = 192;

struct TcArgs {
  CUtensorMap mapA[3];
  CUtensorMap mapB;
  int seg_rows[3];
  int nseg;
  int swiglu;
  int M, K, KB, NT, n_wtiles, n_ttiles;
  long long units;
  int stages;
  int epi;
  float* out;
  int ldo;
  bf16* out_bf;
  int ldh;
  const float* bias;
  int ld_bias;
  const int* row_seq;
  int sp;            // CTAs per tile (cluster size); 1 = whole tiles, persistent
  int tiles;
  unsigned* err;
  unsigned long long* stamp;   // in-graph timing (GemmArgs::stamp), may be null
  // EPI_QKV
  float* q_out;
  bf16* kv_pool;
  const int* kv_table;
  int kv_bt_stride, kv_n_blocks, n_heads, n_kv_heads, head_dim, layer;
  const float* rope_cs;
  const int* row_pos;
  const int* row_valid;
  // fused RMSNorm (see GemmArgs)
  const bf16* norm_gamma;
  bf16* norm_out;
  float* norm_ssq_out;
  float* tap;
  const int* tap_row;
  int tap_mask;
  const float* norm_ssq_in;
  int norm_parts, norm_d;
  float norm_eps;
  int ld_ssq;
  // fused decode attention (see GemmArgs)
  const float* attn_q;
  const int* attn_seq;
  const int* attn_pre_len;
  int attn_pre_stable, attn_pre_fresh;
};


// The kernel's arguments with the epilogue kind fixed at compile time: epi and swiglu hide the
// base's run-time fields, so each instantiation of the kernel (one per epilogue) carries only its
// own epilogue's code.
template <int E>
struct TcArgsE : TcArgs {
  static constexpr int epi = E;
  static constexpr int swiglu = E == EPI_SWIGLU ? 1 : 0;
};

constexpr int kMaxNT = 256;  // token columns per tile

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
constexpr int kXS = 17;   // padded row of the epilogue exchange buffer (128 rows x 16 columns)

// ------------------------------------------------------------------------------ epilogue stores
// One output value of weight row `row` of tile (wt, tt) for token m (m < M).
__device__ __forceinline__ float add_bias_of(const TcArgs& a, int n, int m) {
  return a.bias ? a.bias[static_cast<size_t>(a.row_seq ? a.row_seq[m] : 0) * a.ld_bias + n] : 0.f;
}
__device__ __forceinline__ float silu_f(float y) { return y / (1.f + __expf(-y)); }
template <class A>
__device__ __forceinline__ void emit_plain(const A& a, int wt, int row, int m, float v) {
  const int n = wt * kWRows + row;
  if (a.epi == EPI_SILU) {
    a.out_bf[static_cast<size_t>(m) * a.ldh + n] = __float2bfloat16_rn(silu_f(v + add_bias_of(a, n, m)));
    return;
  }
  float* o = a.out + static_cast<size_t>(m) * a.ldo + n;
  if (a.epi == EPI_ADD) *o += v + add_bias_of(a, n, m);
  else *o = v;
}
// Eq. 2 for feature f of the tile (gate row f, up row f + 64).
__device__ __forceinline__ void emit_swiglu(const TcArgs& a, int wt, int f, int m, float gate, float up) {
  const int feat = wt * 64 + f;
  if (a.bias) up += a.bias[static_cast<size_t>(a.row_seq ? a.row_seq[m] : 0) * a.ld_bias + feat];
  a.out_bf[static_cast<size_t>(m) * a.ldh + feat] = __float2bfloat16_rn(up * (gate / (1.f + __expf(-gate))));
}
// Tile rows are whole heads of [q | k | v]; q and k are rotated with their rotate-half partner
// (row +- hd/2 of the same head), q goes to q_out and k, v of valid rows to the paged cache.
__device__ __forceinline__ void emit_qkv(const TcArgs& a, int wt, int row, int m, float v, float vp) {
  const int hd = a.head_dim, half = hd >> 1;
  const int n = wt * kWRows + row;
  const int head = n / hd, i = n % hd;
  const int pos = a.row_pos[m];
  float o = v;
  if (head < a.n_heads + a.n_kv_heads) {
    const int ir = (i < half) ? i : i - half;
    const float2 cs = reinterpret_cast<const float2*>(a.rope_cs)[static_cast<size_t>(pos) * half + ir];
    o = (i < half) ? v * cs.x - vp * cs.y : v * cs.x + vp * cs.y;
  }
  if (head < a.n_heads) {
    a.q_out[(static_cast<size_t>(m) * a.n_heads + head) * hd + i] = o;
  } else if (a.row_valid[m]) {
    const int kvi = (head - a.n_heads) / a.n_kv_heads;            // 0: K, 1: V
    const int kvh = (head - a.n_heads) % a.n_kv_heads;
    const int blk = a.kv_table[static_cast<size_t>(a.row_seq[m]) * a.kv_bt_stride + (pos >> 4)];
    a.kv_pool[((static_cast<size_t>(a.layer) * a.kv_n_blocks + blk) * 2 + kvi) * a.n_kv_heads * 16 * hd +
              static_cast<size_t>(kvh) * 16 * hd + (pos & 15) * hd + i] = __float2bfloat16_rn(o);
  }
}
__device__ __forceinline__ int partner_row(const TcArgs& a, int row) {
  const int half = a.head_dim >> 1;
  return ((row % a.head_dim) < half) ? row + half : row - half;
}

// Fused RMSNorm, producer side: the updated residual x_new of output (token m, feature n) also
// goes out as bf16(x_new * gamma[n]) and, for tap rows, into the tap slots.
__device__ __forceinline__ void norm_produce(const TcArgs& a, int m, int n, float xn, float g) {
  a.norm_out[static_cast<size_t>(m) * a.ldo + n] = __float2bfloat16_rn(xn * g);
  if (a.tap_mask) {
    const int tr = a.tap_row ? a.tap_row[m] : m;
    if (tr >= 0)
      for (int s = 0; s < 3; ++s)
        if (a.tap_mask & (1 << s)) a.tap[(static_cast<size_t>(tr) * 3 + s) * a.ldo + n] = xn;
  }
}
// Fused RMSNorm, consumer side: rs[c] = rsqrt(mean of x_new^2 + eps) of the token tile's columns,
// from the producer's slices summed in a fixed order (8 strided partial sums, then a butterfly
// over the 8 lanes). Called by the 128 epilogue threads (tid = 0..127). Each lane requests its
// slices in blocks of 32 before adding any (indices clamped), so a block costs one L2 round trip.
__device__ __forceinline__ void tile_rstd(const TcArgs& a, int tt, float* rs, int tid) {
  const int cols = min(a.NT, a.M - tt * a.NT);
  const int j = tid & 7;
  for (int c0 = 0; c0 < cols; c0 += 16) {
    const int c = c0 + (tid >> 3);
    float s = 0.f;
    if (c < cols) {
      const float* src = a.norm_ssq_in + tt * a.NT + c;
      for (int p0 = j; p0 < a.norm_parts; p0 += 8 * 32) {
        float v[32];
#pragma unroll
        for (int u = 0; u < 32; ++u) v[u] = src[static_cast<size_t>(min(p0 + 8 * u, a.norm_parts - 1)) * a.ld_ssq];
#pragma unroll
        for (int u = 0; u < 32; ++u) s = p0 + 8 * u < a.norm_parts ? s + v[u] : s;
      }
    }
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 4);
    if (j == 0 && c < cols) rs[c] = rsqrtf(s / static_cast<float>(a.norm_d) + a.norm_eps);
  }
}

// Whole-tile epilogue: thread r holds weight row r for 16 token columns j0..j0+15; rows that
// need another row (SwiGLU pairs, rotate-half partners) are exchanged through shared memory.
template <class A>
__device__ __forceinline__ void finish_chunk(const A& a, int wt, int tt, int r, int j0, float (&v)[16],
                                             float* xbuf, const float* rs) {
  const int m0 = tt * a.NT + j0;
  if (a.norm_ssq_in)
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] *= rs[j0 + j];
  if (a.epi == EPI_QKV || a.swiglu) {
#pragma unroll
    for (int j = 0; j < 16; ++j) xbuf[r * kXS + j] = v[j];
    named_bar_epi();
    if (a.swiglu) {
      if (r < 64)
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (m0 + j < a.M) emit_swiglu(a, wt, r, m0 + j, v[j], xbuf[(r + 64) * kXS + j]);
    } else {
      const int p = partner_row(a, r);
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (m0 + j < a.M) emit_qkv(a, wt, r, m0 + j, v[j], xbuf[p * kXS + j]);
    }
    named_bar_epi();
    return;
  }
  if (a.norm_out) {
    // residual add, bf16(x_new * gamma), taps, and this tile's sums of squares per token
    const int n = wt * kWRows + r;
    const float g = __bfloat162float(a.norm_gamma[n]);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float sq = 0.f;
      if (m0 + j < a.M) {
        float* o = a.out + static_cast<size_t>(m0 + j) * a.ldo + n;
        const float xn = *o + (v[j] + add_bias_of(a, n, m0 + j));
        *o = xn;
        norm_produce(a, m0 + j, n, xn, g);
        sq = xn * xn;
      }
      xbuf[r * kXS + j] = sq;
    }
    named_bar_epi();
    const int jj = r >> 3, sg = r & 7;   // column jj, rows 16 sg .. 16 sg + 15
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) s += xbuf[(sg * 16 + i) * kXS + jj];
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 4);
    if (sg == 0 && m0 + jj < a.M) a.norm_ssq_out[static_cast<size_t>(wt) * a.ld_ssq + m0 + jj] = s;
    named_bar_epi();
    return;
  }
#pragma unroll
  for (int j = 0; j < 16; ++j)
    if (m0 + j < a.M) emit_plain(a, wt, r, m0 + j, v[j]);
}

// Split-K pairs: the 128 rows of a tile as 64 pairs whose members one epilogue needs together.
// SwiGLU: (gate f, up f) = rows (p, p + 64); QKV with hd = 128: rotate-half partners (i, i + 64);
// QKV with hd = 64 (two heads per tile): (64h + i, 64h + i + 32); plain outputs: (p, p + 64).
template <class A>
__device__ __forceinline__ bool pairs_of_32(const A& a) { return a.epi == EPI_QKV && a.head_dim == 64; }
template <class A>
__device__ __forceinline__ int pair_of(const A& a, int row) {
  return pairs_of_32(a) ? (row >> 6) * 32 + (row & 31) : (row & 63);
}
template <class A>
__device__ __forceinline__ int member_of(const A& a, int row) {
  return pairs_of_32(a) ? ((row >> 5) & 1) : (row >> 6);
}
template <class A>
__device__ __forceinline__ int pair_row(const A& a, int p, int m) {
  return pairs_of_32(a) ? (p >> 5) * 64 + m * 32 + (p & 31) : p + 64 * m;
}
// Rank r of sp owns pairs [64 r / sp, 64 (r + 1) / sp); its receive buffer holds, per source
// rank q and owned pair lp, both members' NT columns: [q][lp][member][NT] floats. Within a row
// the 16-byte chunks of four columns are rotated by lp mod 8 (recv_chunk), so the owner's reads
// of one column across consecutive pairs fall in different bank groups: unrotated, every row
// starts at the same bank (2 NT is a multiple of 32 words) and such a read is np-way conflicted.
__device__ __forceinline__ int pair_owner(int p, int sp) { return ((p + 1) * sp - 1) / 64; }
__device__ __forceinline__ int pairs_max(int sp) { return (64 + sp - 1) / sp; }
__device__ __forceinline__ int recv_chunk(int c4, int lp, int nch) {   // nch = NT / 4, a multiple of 4
  int rot = lp & 7;
  rot = rot >= nch ? rot - nch : rot;
  const int x = c4 + rot;
  return x >= nch ? x - nch : x;
}

// The global operands of one output pair (pair p of tile wt, token m), loaded before its sums
// are known: residuals (EPI_ADD), steering bias (SwiGLU), or position, rotary factors and KV
// block (QKV; blk = -1 when the pair is a q head or the row writes no KV).
struct PairOps {
  float r0, r1, bias, bias1, g0, g1;   // bias: SwiGLU's, or EPI_ADD's for member 0 (bias1: member 1)
  float2 cs;
  int pos, blk;
};
template <class A>
__device__ __forceinline__ PairOps pair_ops(const A& a, int wt, int p, int m) {
  PairOps o{0.f, 0.f, 0.f, 0.f, 0.f, 0.f, make_float2(1.f, 0.f), 0, -1};
  if (a.swiglu) {
    if (a.bias) o.bias = a.bias[static_cast<size_t>(a.row_seq ? a.row_seq[m] : 0) * a.ld_bias + wt * 64 + p];
  } else if (a.epi == EPI_QKV) {
    const int hd = a.head_dim, half = hd >> 1;
    const int n = wt * kWRows + pair_row(a, p, 0);
    const int head = n / hd, i = n % hd;
    o.pos = a.row_pos[m];
    if (head < a.n_heads + a.n_kv_heads)
      o.cs = reinterpret_cast<const float2*>(a.rope_cs)[static_cast<size_t>(o.pos) * half + i];
    if (head >= a.n_heads && a.row_valid[m])
      o.blk = a.kv_table[static_cast<size_t>(a.row_seq[m]) * a.kv_bt_stride + (o.pos >> 4)];
  } else if (a.epi == EPI_SILU) {
    o.bias = add_bias_of(a, wt * kWRows + pair_row(a, p, 0), m);
    o.bias1 = add_bias_of(a, wt * kWRows + pair_row(a, p, 1), m);
  } else if (a.epi == EPI_ADD) {
    const float* x = a.out + static_cast<size_t>(m) * a.ldo + wt * kWRows;
    o.r0 = x[pair_row(a, p, 0)];
    o.r1 = x[pair_row(a, p, 1)];
    o.bias = add_bias_of(a, wt * kWRows + pair_row(a, p, 0), m);
    o.bias1 = add_bias_of(a, wt * kWRows + pair_row(a, p, 1), m);
    if (a.norm_out) {
      o.g0 = __bfloat162float(a.norm_gamma[wt * kWRows + pair_row(a, p, 0)]);
      o.g1 = __bfloat162float(a.norm_gamma[wt * kWRows + pair_row(a, p, 1)]);
    }
  }
  return o;
}
// Epilogue of one output pair from its split-K sums s0 (member 0) and s1 (member 1). Returns the
// pair's contribution to the token's sum of squares when it produces a fused RMSNorm.
template <class A>
__device__ __forceinline__ float pair_emit(const A& a, int wt, int p, int m, float s0, float s1, const PairOps& o) {
  if (a.swiglu) {
    const float up = s1 + o.bias;
    a.out_bf[static_cast<size_t>(m) * a.ldh + wt * 64 + p] = __float2bfloat16_rn(up * (s0 / (1.f + __expf(-s0))));
  } else if (a.epi == EPI_QKV) {
    // members are rotate-half partners i < hd/2 and i + hd/2 of one head
    const int hd = a.head_dim, half = hd >> 1;
    const int n = wt * kWRows + pair_row(a, p, 0);
    const int head = n / hd, i = n % hd;
    float o0 = s0, o1 = s1;
    if (head < a.n_heads + a.n_kv_heads) {
      o0 = s0 * o.cs.x - s1 * o.cs.y;
      o1 = s1 * o.cs.x + s0 * o.cs.y;
    }
    if (head < a.n_heads) {
      float* q = a.q_out + (static_cast<size_t>(m) * a.n_heads + head) * hd;
      q[i] = o0;
      q[i + half] = o1;
    } else if (o.blk >= 0) {
      const int kvi = (head - a.n_heads) / a.n_kv_heads;            // 0: K, 1: V
      const int kvh = (head - a.n_heads) % a.n_kv_heads;
      bf16* dst = a.kv_pool + ((static_cast<size_t>(a.layer) * a.kv_n_blocks + o.blk) * 2 + kvi) * a.n_kv_heads * 16 * hd +
                  static_cast<size_t>(kvh) * 16 * hd + (o.pos & 15) * hd;
      dst[i] = __float2bfloat16_rn(o0);
      dst[i + half] = __float2bfloat16_rn(o1);
    }
  } else if (a.epi == EPI_SILU) {
    bf16* hb = a.out_bf + static_cast<size_t>(m) * a.ldh + wt * kWRows;
    hb[pair_row(a, p, 0)] = __float2bfloat16_rn(silu_f(s0 + o.bias));
    hb[pair_row(a, p, 1)] = __float2bfloat16_rn(silu_f(s1 + o.bias1));
  } else {
    float* x = a.out + static_cast<size_t>(m) * a.ldo + wt * kWRows;
    const bool add = a.epi == EPI_ADD;
    const float x0 = add ? o.r0 + (s0 + o.bias) : s0, x1 = add ? o.r1 + (s1 + o.bias1) : s1;
    x[pair_row(a, p, 0)] = x0;
    x[pair_row(a, p, 1)] = x1;
    if (a.norm_out) {
      norm_produce(a, m, wt * kWRows + pair_row(a, p, 0), x0, o.g0);
      norm_produce(a, m, wt * kWRows + pair_row(a, p, 1), x1, o.g1);
      return x0 * x0 + x1 * x1;
    }
  }
  return 0.f;
}


// Shared memory and launch facts the split-K epilogue needs.
struct SplitK {
  unsigned char* smem;                       // the drained ring: fused-norm scratch
  float* recv;                               // [sp][npmax][2][NT] partials of this rank's pairs
  float* rs;                                 // RMSNorm row scales (consumers)
  volatile int* flags;
  uint32_t tfull0, rbar, tmem;
  int rank, sp, npmax, NT, first_tile;
};
// The global operands of the first output this epilogue thread (tid 0..127) owns, fetched early.
template <class A>
__device__ __forceinline__ PairOps first_pair_ops(const A& a, int rank, int sp, int NT, int first_tile, int tid) {
  const int wt = first_tile % a.n_wtiles, tt = first_tile / a.n_wtiles;
  const int cols = min(NT, a.M - tt * NT);
  const int p_lo = rank * 64 / sp, np = (rank + 1) * 64 / sp - p_lo;
  return tid < np * cols && np * cols <= 128 ? pair_ops(a, wt, p_lo + tid % np, tt * NT + tid / np) : PairOps{};
}
// Sum in rank order of the sp partials of one receive-buffer word (T = float) or four adjacent
// ones (T = float4); rv points at rank 0's member-0 value, member 1 is NT floats on, rank q at q
// rstride floats. C >= sp loads per member are issued before any add (rank index clamped).
__device__ __forceinline__ void add_part(float& s, float v) { s += v; }
__device__ __forceinline__ void add_part(float4& s, float4 v) { s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w; }
template <int C, typename T>
__device__ __forceinline__ void sum_parts(const float* rv, int rstride, int NT, int sp, T& s0, T& s1) {
  T v0[C], v1[C];
#pragma unroll
  for (int j = 0; j < C; ++j) {
    const int kk = min(j, sp - 1);
    v0[j] = *reinterpret_cast<const T*>(rv + kk * rstride);
    v1[j] = *reinterpret_cast<const T*>(rv + kk * rstride + NT);
  }
  s0 = v0[0];
  s1 = v1[0];
#pragma unroll
  for (int j = 1; j < C; ++j)
    if (j < sp) {
      add_part(s0, v0[j]);
      add_part(s1, v1[j]);
    }
}
template <typename T>
__device__ __forceinline__ void sum_parts_any(const float* rv, int rstride, int NT, int sp, T& s0, T& s1) {
  if (sp <= 2) sum_parts<2>(rv, rstride, NT, sp, s0, s1);
  else if (sp <= 4) sum_parts<4>(rv, rstride, NT, sp, s0, s1);
  else sum_parts<8>(rv, rstride, NT, sp, s0, s1);
}
// Split-K epilogue of the CTA's single tile (sp > 1), run by the four epilogue warps (warp % 4 =
// the TMEM lane quarter): this rank's partial of every row goes to the rank owning the row's pair
// (st.async onto the owner's receive barrier); the owner waits for its own pairs only, sums the
// partials in rank order and runs the epilogue. Everything but the sums is prepared while the
// MMAs run. pf: the operands of the thread's first owned output (first_pair_ops).
template <class A>
__device__ __forceinline__ void splitk_epilogue(const A& a, const SplitK& sk, int warp, int lane, const PairOps& pf) {
  const int q = warp & 3, r = q * 32 + lane, tid = threadIdx.x - 64;
  const bool leader = (warp == 2 && lane == 0);
  const int sp = sk.sp, npmax = sk.npmax, NT = sk.NT, rank = sk.rank;
  volatile int* flags = sk.flags;
  volatile int* abort_flag = sk.flags;
  float* recv = sk.recv;
  float* rs = sk.rs;
  const int wt = sk.first_tile % a.n_wtiles, tt = sk.first_tile / a.n_wtiles;
  const int cols = min(NT, a.M - tt * NT);
  const int p_lo = rank * 64 / sp, np = (rank + 1) * 64 / sp - p_lo;
  const int p = pair_of(a, r), owner = pair_owner(p, sp), lpd = p - owner * 64 / sp, nch = NT >> 2;
  const int slot = ((rank * npmax + lpd) * 2 + member_of(a, r)) * NT;
  const uint32_t dst = dsmem_addr(smem_u32(recv + slot), static_cast<uint32_t>(owner));
  const uint32_t dst_bar = dsmem_addr(sk.rbar, static_cast<uint32_t>(owner));
  if (a.norm_ssq_in) tile_rstd(a, tt, rs, tid);
  cluster_wait();                          // every rank's receive barrier is armed (every thread of the
                                           // cluster arrived at kernel start: taken while the MMAs run)
  if (leader) flags[4] = wait_bar(sk.tfull0, 0, abort_flag, a.err) ? 1 : 0;
  named_bar_epi();                         // the accumulator is complete (or the wait gave up); rs is set
  tc_fence_after();
  if (flags[4] != 0) {
    const uint32_t tbase = sk.tmem + (static_cast<uint32_t>(q * 32) << 16);
    for (int ch = 0; ch * 16 < cols; ++ch) {
      float v[16];
      tmem_ld16(tbase + ch * 16, v);
#pragma unroll
      for (int k4 = 0; k4 < 4; ++k4)
        st_async_v4(dst + static_cast<uint32_t>(recv_chunk(ch * 4 + k4, lpd, nch) * 16), dst_bar, v[4 * k4],
                    v[4 * k4 + 1], v[4 * k4 + 2], v[4 * k4 + 3]);
    }
    if (leader) flags[5] = wait_bar(sk.rbar, 0, abort_flag, a.err) ? 1 : 0;
    named_bar_epi();
    if (flags[5] != 0) {
      // every rank's partial of this rank's pairs is in the receive buffer: sums in rank order
      float* sq = reinterpret_cast<float*>(sk.smem);   // [cols][np] fused-norm sums of squares (drained ring)
      const int rstride = npmax * 2 * NT, n_own = np * cols;
      if (n_own <= 128) {
        // one output per thread, whose operands were fetched while the MMAs ran
        const int e = tid;
        if (e < n_own) {
          const int lp = e % np, col = e / np;
          float s0, s1;
          sum_parts_any(recv + lp * 2 * NT + recv_chunk(col >> 2, lp, nch) * 4 + (col & 3), rstride, NT, sp, s0, s1);
          if (a.norm_ssq_in) {
            s0 *= rs[col];
            s1 *= rs[col];
          }
          const float q2 = pair_emit(a, wt, p_lo + lp, tt * NT + col, s0, s1, pf);
          if (a.norm_out) sq[col * np + lp] = q2;
        }
      } else {
        // wide token tiles: a thread takes pair lp over four adjacent columns, reads their
        // partials as 16-byte words (one rotated chunk) and requests all four outputs' global
        // operands before it stores any, so each pass costs one memory round trip, not four
        const int nq = np * ((cols + 3) >> 2);
        for (int e = tid; e < nq; e += 128) {
          const int lp = e % np, c4 = e / np;
          PairOps o[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) o[u] = pair_ops(a, wt, p_lo + lp, tt * NT + min(4 * c4 + u, cols - 1));
          float4 s0, s1;
          sum_parts_any(recv + lp * 2 * NT + recv_chunk(c4, lp, nch) * 4, rstride, NT, sp, s0, s1);
          const float v0[4] = {s0.x, s0.y, s0.z, s0.w}, v1[4] = {s1.x, s1.y, s1.z, s1.w};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int col = 4 * c4 + u;
            if (col < cols) {
              const float sc = a.norm_ssq_in ? rs[col] : 1.f;
              const float q2 = pair_emit(a, wt, p_lo + lp, tt * NT + col, a.norm_ssq_in ? v0[u] * sc : v0[u],
                                         a.norm_ssq_in ? v1[u] * sc : v1[u], o[u]);
              if (a.norm_out) sq[col * np + lp] = q2;
            }
          }
        }
      }
      if (a.norm_out) {   // this rank's slice of the tile: sums of squares per token, in pair order
        named_bar_epi();
        for (int c = tid; c < cols; c += 128) {
          float ssum = 0.f;
          for (int lp = 0; lp < np; ++lp) ssum += sq[c * np + lp];
          a.norm_ssq_out[static_cast<size_t>(wt * sp + rank) * a.ld_ssq + tt * NT + c] = ssum;
        }
      }
    } else if (leader) {
      wait_bar_budget(sk.rbar, 0, kDrainCycles);   // let partials still in flight land before leaving
    }
  } else if (leader) {
    // This rank's accumulator never completed (a wait gave up), so it pushes nothing; the other
    // ranks push their partials of its pairs right after their own accumulators, with no wait in
    // between, and may still be doing so: let them land before the CTA (and its shared memory)
    // goes away. Every rank reaches its pushes, or skips them, within the bounded waits above.
    wait_bar_budget(sk.rbar, 0, kDrainCycles);
  }
}

// SPLIT: 1 = every launch of this instantiation splits K (sp > 1), 2 = whole tiles (sp == 1),
// 0 = decided at run time.
template <class A, int SPLIT>
__global__ void __launch_bounds__(kThreads, 2) gemm_tc_kernel(const __grid_constant__ A a) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = a.stages, NT = a.NT, sp = SPLIT == 2 ? 1 : a.sp;
  const bool split = SPLIT == 1 ? true : (SPLIT == 2 ? false : sp > 1);
  const uint32_t a_bytes = kWRows * kBK * 2;
  const uint32_t b_bytes = static_cast<uint32_t>(NT) * kBK * 2;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  const int npmax = pairs_max(sp);
  const uint32_t recv_bytes = split ? static_cast<uint32_t>(sp * npmax * 2 * NT * 4) : 0u;
  float* recv = reinterpret_cast<float*>(smem + static_cast<size_t>(S) * stage_bytes);  // split-K partials in
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(S) * stage_bytes + recv_bytes);
  // bars: full[S], empty[S], tfull[2], tempty[2], drain, recv (split-K partials of this rank's pairs)
  float* xbuf = reinterpret_cast<float*>(bars + 2 * S + 6);
  volatile int* flags = reinterpret_cast<volatile int*>(xbuf + kWRows * kXS);
  // flags: [0] abort, [1] TMEM base, [3] stages consumed, [4] go, [5] partials received
  float* rs = const_cast<float*>(reinterpret_cast<volatile float*>(flags + 16));   // [kMaxNT] fused-norm scales
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, tfull0 = empty0 + 8 * S, tempty0 = tfull0 + 16,
                 drain = tempty0 + 16, rbar = drain + 8;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t ncols = 32;
  // two accumulators (double buffering) only for a CTA that takes several whole tiles
  const bool one_acc = split || a.tiles <= static_cast<int>(gridDim.x);
  while (ncols < static_cast<uint32_t>((one_acc ? 1 : 2) * NT)) ncols <<= 1;
  const int rank = split ? static_cast<int>(cluster_rank()) : 0;
  if (a.stamp && threadIdx.x == 0) atomicMin(&a.stamp[0], global_ns());

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(tfull0, 1);
    mbar_init(tfull0 + 8, 1);
    mbar_init(tempty0, 4);
    mbar_init(tempty0 + 8, 4);
    mbar_init(drain, 1);
    if (split) {
      // Split-K: every rank pushes its partial of each row to the rank owning the row's pair;
      // the owner's receive barrier completes when all sp partials of its pairs have landed:
      // sp x (2 rows x its pairs) x 64 bytes per 16 token columns.
      const int np = (rank + 1) * 64 / sp - rank * 64 / sp;
      const int cols = min(NT, a.M - (static_cast<int>(blockIdx.x) / sp / a.n_wtiles) * NT);
      mbar_init(rbar, 1);
      mbar_expect_tx(rbar, static_cast<uint32_t>(sp * 2 * np * ((cols + 15) / 16) * 64));
    }
    flags[0] = 0; flags[3] = 0; flags[4] = 0; flags[5] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<int*>(flags) + 1), ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (split) cluster_arrive_relaxed();      // waited for before the first push into another rank
  const uint32_t tmem = static_cast<uint32_t>(flags[1]);
  volatile int* abort_flag = flags;

  // This CTA's segments: sp > 1 -> one K-slice of tile blockIdx.x / sp; sp == 1 -> whole tiles
  // blockIdx.x, blockIdx.x + gridDim.x, ...
  const int first_tile = split ? static_cast<int>(blockIdx.x) / sp : static_cast<int>(blockIdx.x);
  const int tile_step = split ? a.tiles : static_cast<int>(gridDim.x);
  const int kb_lo = rank * a.KB / sp, kb_hi = (rank + 1) * a.KB / sp;
  const int nkb = kb_hi - kb_lo;

  pdl_trigger();                             // the next kernel may start its own prologue
  PairOps pf{};                              // split-K: operands of this thread's first output pair
  if (warp == 0) {
    // Stage use j loads k-block (kb_lo + j % nkb) of the CTA's (j / nkb)-th tile: the weight half
    // first, then the token half. Weights never depend on earlier kernels, so the first stages'
    // weight tiles are requested before waiting for the predecessor grid. Cursors advance one
    // k-block at a time (no divisions in the issue loop).
    struct Cursor {
      int tile, kb, wt, tt, seg, row0;
    };
    auto locate = [&](Cursor& c) {
      c.wt = c.tile % a.n_wtiles;
      c.tt = c.tile / a.n_wtiles;
      c.seg = 0;
      c.row0 = c.wt * kWRows;
      if (!a.swiglu)
        while (c.seg + 1 < a.nseg && c.row0 >= a.seg_rows[c.seg]) c.row0 -= a.seg_rows[c.seg++];
    };
    auto advance = [&](Cursor& c) {
      if (++c.kb == kb_hi) { c.kb = kb_lo; c.tile += tile_step; if (c.tile < a.tiles) locate(c); }
    };
    int n_my_tiles = 0;
    for (int t = first_tile; t < a.tiles; t += tile_step) ++n_my_tiles;
    const uint32_t n_units = static_cast<uint32_t>(n_my_tiles * nkb);
    const uint64_t wpol = l2_evict_first();
    Cursor ca;
    ca.tile = first_tile;
    ca.kb = kb_lo;
    if (ca.tile < a.tiles) locate(ca);
    auto load_a = [&](uint32_t s, const Cursor& c) {   // into stage s
      const uint32_t dst = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
      if (a.swiglu) {
        tma_load_2d_stream(dst, &a.mapA[0], c.kb * kBK, c.wt * 64, full0 + 8 * s, wpol);
        tma_load_2d_stream(dst + a_bytes / 2, &a.mapA[1], c.kb * kBK, c.wt * 64, full0 + 8 * s, wpol);
      } else {
        tma_load_2d_stream(dst, &a.mapA[c.seg], c.kb * kBK, c.row0, full0 + 8 * s, wpol);
      }
    };
    auto load_b = [&](uint32_t s, const Cursor& c) {
      const uint32_t dst = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
      tma_load_2d(dst + a_bytes, &a.mapB, c.kb * kBK, c.tt * NT, full0 + 8 * s);
    };
    const uint32_t pre = n_units < static_cast<uint32_t>(S) ? n_units : static_cast<uint32_t>(S);
    if (lane == 0)
      for (uint32_t j = 0; j < pre; ++j, advance(ca)) {   // first use of each stage: no wait
        mbar_expect_tx(full0 + 8 * j, stage_bytes);
        load_a(j, ca);
      }
    __syncwarp();                            // the stages' expected bytes are set before any token load
    pdl_wait();
    if (lane == 0 && a.stamp) atomicMin(&a.stamp[1], global_ns());
    // The token halves of the first stages, one lane each: one issue instead of `pre` in a row
    // (each TMA issue takes a few hundred cycles).
    if (lane < pre) {
      Cursor cb;
      cb.tile = first_tile + static_cast<int>(lane / static_cast<uint32_t>(nkb)) * tile_step;
      cb.kb = kb_lo + static_cast<int>(lane % static_cast<uint32_t>(nkb));
      locate(cb);
      tma_load_2d(smem_u32(smem + static_cast<size_t>(lane) * stage_bytes) + a_bytes, &a.mapB, cb.kb * kBK,
                  cb.tt * NT, full0 + 8 * lane);
    }
    __syncwarp();
    if (lane == 0) {
      uint32_t j = pre;
      uint32_t s = pre % static_cast<uint32_t>(S), ph = (pre / static_cast<uint32_t>(S)) & 1;   // stage of use j, its phase
      bool ok = true;
      for (; j < n_units; ++j, advance(ca)) {
        if (!wait_bar(empty0 + 8 * s, ph ^ 1, abort_flag, a.err)) { ok = false; break; }
        mbar_expect_tx(full0 + 8 * s, stage_bytes);
        load_a(s, ca);
        load_b(s, ca);
        if (++s == static_cast<uint32_t>(S)) { s = 0; ph ^= 1u; }
      }
      if (!ok) {  // let the loads already issued land before the CTA exits
        const uint32_t done = static_cast<uint32_t>(flags[3]);
        for (uint32_t jj = done; jj < j; ++jj) wait_bar_budget(full0 + 8 * (jj % S), (jj / S) & 1, kDrainCycles);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kWRows, NT);
      // stage s of use j = j mod S and its phase, advanced incrementally; a stage's descriptors are
      // the ring base's plus the stage offset (the address field is addr >> 4, below 2^14)
      const uint64_t desc0 = sw128_desc(smem_u32(smem));
      const uint64_t dstage = stage_bytes >> 4, dB = a_bytes >> 4;
      // With every stage used once (all of the CTA's k-blocks fit the ring) the producer never
      // waits for a stage to drain: no per-stage release, and nothing for its abort path to count.
      int n_my_tiles = 0;
      for (int t = first_tile; t < a.tiles; t += tile_step) ++n_my_tiles;
      const bool reuse = n_my_tiles * nkb > S;
      uint32_t j = 0, segi = 0, s = 0, ph = 0;
      bool ok = true;
      for (int t = first_tile; t < a.tiles && ok; t += tile_step, ++segi) {
        const uint32_t acc = segi & 1;
        if (!wait_bar(tempty0 + 8 * acc, ((segi >> 1) & 1) ^ 1, abort_flag, a.err)) break;
        tc_fence_after();
        const uint32_t d = tmem + acc * NT;
        for (int i = 0; i < nkb; ++i, ++j) {
          if (!wait_bar(full0 + 8 * s, ph, abort_flag, a.err)) { ok = false; break; }
          tc_fence_after();
          const uint64_t ad = desc0 + s * dstage, bd = ad + dB;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            mma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
          if (reuse) {
            mma_commit(empty0 + 8 * s);
            flags[3] = static_cast<int>(j + 1);
          }
          if (++s == static_cast<uint32_t>(S)) { s = 0; ph ^= 1u; }
        }
        if (!ok) break;
        mma_commit(tfull0 + 8 * acc);
      }
      mma_commit(drain);                      // all MMAs issued by this thread have completed
      wait_bar_budget(drain, 0, kDrainCycles);
    }
  } else if (split) {
    // Split-K epilogue of the CTA's single tile. Everything but the sums (this thread's
    // destination in the owner's receive buffer, the operands of its first owned output, the
    // RMSNorm scales) is prepared while the MMAs run.
    pdl_wait();                              // outputs, residuals and biases come from earlier kernels
    pf = first_pair_ops(a, rank, sp, NT, first_tile, threadIdx.x - 64);
    splitk_epilogue(a, SplitK{smem, recv, rs, flags, tfull0, rbar, tmem, rank, sp, npmax, NT, first_tile}, warp, lane, pf);
  } else {
    const int q = warp & 3;                   // TMEM lane quarter of this warp
    const int r = q * 32 + lane;              // weight row within the tile
    const bool leader = (warp == 2 && lane == 0);
    pdl_wait();                              // outputs, residuals and biases come from earlier kernels
    uint32_t segi = 0;
    int rs_tt = -1;
    for (int t = first_tile; t < a.tiles; t += tile_step, ++segi) {
      const uint32_t acc = segi & 1;
      const int wt = t % a.n_wtiles, tt = t / a.n_wtiles;
      if (a.norm_ssq_in && tt != rs_tt) {    // RMSNorm scales of the token tile, while its MMAs run
        named_bar_epi();                     // no thread still reads the previous tile's scales
        tile_rstd(a, tt, rs, threadIdx.x - 64);
        rs_tt = tt;
      }
      if (leader) flags[4] = wait_bar(tfull0 + 8 * acc, (segi >> 1) & 1, abort_flag, a.err) ? 1 : 0;
      named_bar_epi();
      const bool go = flags[4] != 0;
      tc_fence_after();
      if (!go) break;
      const uint32_t tbase = tmem + (static_cast<uint32_t>(q * 32) << 16) + acc * NT;
      const int cols = min(NT, a.M - tt * NT);   // token columns of this tile that exist
      for (int ch = 0; ch * 16 < cols; ++ch) {
        float v[16];
        tmem_ld16(tbase + ch * 16, v);
        finish_chunk(a, wt, tt, r, ch * 16, v, xbuf, rs);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
    }
  }

  if (split && warp < 2) {                  // the producer and MMA warps take their half of the cluster barrier
    __syncwarp();
    cluster_wait();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, ncols);
  if (a.stamp && threadIdx.x == 0) atomicMax(&a.stamp[2], global_ns());
}


// ------------------------------------------------------------------------------ fused decode attention
// The O projection of a decode step of one sequence with its attention folded in. With sp = H_kv
// ranks per tile, rank r's K-slice of W_O is exactly the G = H / H_kv query heads of KV head r
// (hd 64: one k-block per head), so CTA (tile, r) computes the causal attention of KV head r for
// the step's rows over the whole context and writes it, in bf16 and in the 128-byte-swizzled
// K-major layout a TMA load would give, as the token operand of its stages; the MMA and the
// split-K epilogue are those of gemm_tc_kernel. The attention is split over 8 warps by position
// ranges (each a flash-decoding pass with its own running max and sum, K/V staged by cp.async
// three 16-position sub-tiles ahead, no CTA barrier per sub-tile), then merged across the warps.
// The 16 O tiles that share a KV head each recompute it (from L2); what this saves is the
// attention kernel, its cluster merge and one kernel boundary per layer.
constexpr int kAoWarps = 10;                 // 0 TMA, 1 MMA, 2-9 attention (2-5 also the epilogue)
constexpr int kAoThreads = kAoWarps * 32;
constexpr int kAoSub = 16;                   // positions per sub-tile
constexpr int kAoBuf = 3;                    // sub-tiles in flight per warp
constexpr int kAoKS = 64 + 8;                // K/V/Q row stride (bf16), hd 64
constexpr int kAoAS = 64 + 4;                // per-warp partial accumulator row stride (f32)
constexpr int kAoMaxBlk = 32;                // cache blocks (of 16 positions) per warp: context <= 4096
constexpr int kAoWarpBytes = kAoBuf * 2 * kAoSub * kAoKS * 2;   // one warp's K/V buffers

__device__ __forceinline__ void named_bar_attn() { asm volatile("bar.sync 2, 256;" ::: "memory"); }
__device__ __forceinline__ uint32_t ao_ld_u32(const bf16* p) { return *reinterpret_cast<const uint32_t*>(p); }
__device__ __forceinline__ uint32_t ao_pack(float x, float y) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ void ao_cp16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0) : "memory");
}
__device__ __forceinline__ void ao_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void ao_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }
__device__ __forceinline__ void ao_mma(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                       uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ao_ldsm_x2_t(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr) : "memory");
}

// Shared memory of the fused kernel after the GEMM part (ring, receive buffer, barriers, flags):
// Q [16][kAoKS] bf16, row positions [16], per-warp (max, sum) [8][16][2], per-warp block ids
// [8][kAoMaxBlk], per-warp K/V buffers [8][kAoWarpBytes] (then each warp's partial accumulators).
constexpr int kAoQBytes = 16 * kAoKS * 2;
constexpr int kAoAttnBytes = kAoQBytes + 16 * 4 + 8 * 16 * 8 + 8 * kAoMaxBlk * 4 + 8 * kAoWarpBytes;

__global__ void __launch_bounds__(kAoThreads, 1) gemm_attn_kernel(const __grid_constant__ TcArgs a) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = a.stages, NT = a.NT, sp = a.sp;   // S = k-blocks of the slice = G
  const uint32_t a_bytes = kWRows * kBK * 2;
  const uint32_t b_bytes = static_cast<uint32_t>(NT) * kBK * 2;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  const int npmax = pairs_max(sp);
  const uint32_t recv_bytes = static_cast<uint32_t>(sp * npmax * 2 * NT * 4);
  float* recv = reinterpret_cast<float*>(smem + static_cast<size_t>(S) * stage_bytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(S) * stage_bytes + recv_bytes);
  volatile int* flags = reinterpret_cast<volatile int*>(bars + 2 * S + 6);
  float* rs = const_cast<float*>(reinterpret_cast<volatile float*>(flags + 16));
  unsigned char* attn = reinterpret_cast<unsigned char*>(rs + 16);
  bf16* sQ = reinterpret_cast<bf16*>(attn);
  int* sPos = reinterpret_cast<int*>(attn + kAoQBytes);
  float* sML = reinterpret_cast<float*>(sPos + 16);                 // [8 warps][16 rows][max, sum]
  int* sBlk = reinterpret_cast<int*>(sML + 8 * 16 * 2);               // [8 warps][kAoMaxBlk]
  unsigned char* sKV = reinterpret_cast<unsigned char*>(sBlk + 8 * kAoMaxBlk);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, tfull0 = empty0 + 8 * S, tempty0 = tfull0 + 16,
                 drain = tempty0 + 16, rbar = drain + 8;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = static_cast<int>(cluster_rank());
  const int first_tile = static_cast<int>(blockIdx.x) / sp;
  const int wt = first_tile % a.n_wtiles;
  const int M = a.M, G = a.n_heads / a.n_kv_heads, nqv = M * G;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 2);           // the weight tile's bytes + the attention's token operand
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(tfull0, 1);
    mbar_init(tfull0 + 8, 1);
    mbar_init(tempty0, 4);
    mbar_init(tempty0 + 8, 4);
    mbar_init(drain, 1);
    const int np = (rank + 1) * 64 / sp - rank * 64 / sp;
    mbar_init(rbar, 1);
    mbar_expect_tx(rbar, static_cast<uint32_t>(sp * 2 * np * ((M + 15) / 16) * 64));
    flags[0] = 0; flags[3] = 0; flags[4] = 0; flags[5] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<int*>(flags) + 1), 32);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_arrive_relaxed();
  const uint32_t tmem = static_cast<uint32_t>(flags[1]);
  volatile int* abort_flag = flags;
  pdl_trigger();

  PairOps pf{};
  if (warp == 0) {
    if (lane == 0) {   // the K-slice of W_O: S weight tiles, requested before the wait (weights are static)
      const uint64_t wpol = l2_evict_first();
      for (int j = 0; j < S; ++j) {
        mbar_expect_tx(full0 + 8 * j, a_bytes);
        tma_load_2d_stream(smem_u32(smem + static_cast<size_t>(j) * stage_bytes), &a.mapA[0], (rank * S + j) * kBK,
                           wt * kWRows, full0 + 8 * j, wpol);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kWRows, NT);
      bool ok = true;
      for (int j = 0; j < S && ok; ++j) {
        if (!wait_bar(full0 + 8 * j, 0, abort_flag, a.err)) { ok = false; break; }
        tc_fence_after();
        const uint32_t abase = smem_u32(smem + static_cast<size_t>(j) * stage_bytes);
        const uint64_t ad = sw128_desc(abase), bd = sw128_desc(abase + a_bytes);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) mma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (j > 0 || kk > 0) ? 1u : 0u);
        mma_commit(empty0 + 8 * j);
      }
      if (ok) mma_commit(tfull0);
      mma_commit(drain);
      wait_bar_budget(drain, 0, kDrainCycles);
    }
  } else {
    // ---- attention of KV head `rank` for the M rows (warps 2-9) ----
    const int aw = warp - 2, at = threadIdx.x - 64;   // attention warp 0..7, thread 0..255
    const int g8 = lane >> 2, t4 = lane & 3;
    const int Hkv = a.n_kv_heads, kvh = rank;
    const int seq = *a.attn_seq;
    const int len = a.attn_pre_len[seq];
    const int row_end = a.kv_bt_stride * 16;
    const int stable = min(max(0, len + a.attn_pre_stable), row_end);
    const int ctx_hi = min(max(stable, len + a.attn_pre_stable + a.attn_pre_fresh), row_end);
    const int P = ((ctx_hi + 8 * kAoSub - 1) / (8 * kAoSub)) * kAoSub;      // positions per warp
    const int w_lo = aw * P, w_hi = min(w_lo + P, ctx_hi);
    const int nsub_all = w_hi > w_lo ? (w_hi - w_lo + kAoSub - 1) / kAoSub : 0;
    int* blk = sBlk + aw * kAoMaxBlk;
    for (int i = lane; i < (P >> 4) && i < kAoMaxBlk; i += 32) {
      const int b16 = (w_lo >> 4) + i;
      blk[i] = b16 < a.kv_bt_stride ? a.kv_table[static_cast<size_t>(seq) * a.kv_bt_stride + b16] : 0;
    }
    __syncwarp();
    const bf16* layer_base = a.kv_pool + static_cast<size_t>(a.layer) * a.kv_n_blocks * 2 * Hkv * 16 * 64 +
                             static_cast<size_t>(kvh) * 16 * 64;
    const size_t blk_stride = static_cast<size_t>(2) * Hkv * 16 * 64;
    unsigned char* wkv = sKV + static_cast<size_t>(aw) * kAoWarpBytes;
    // rows p in [p_from, p_to) of sub-tile j -> slot j % kAoBuf: loaded below `valid_end`, else zero
    auto issue = [&](int j, int p_from, int p_to, int valid_end) {
      bf16* dK = reinterpret_cast<bf16*>(wkv + (j % kAoBuf) * 2 * kAoSub * kAoKS * 2);
      bf16* dV = dK + kAoSub * kAoKS;
      const int t0 = w_lo + j * kAoSub;
#pragma unroll
      for (int u = 0; u < kAoSub * 8 / 32; ++u) {
        const int idx = lane + 32 * u, t = idx >> 3, c = idx & 7;
        const int p = t0 + t;
        if (p < p_from || p >= p_to) continue;
        const bool ok = p < valid_end;
        const bf16* src = layer_base;
        if (ok) src += static_cast<size_t>(blk[(p - w_lo) >> 4]) * blk_stride + static_cast<size_t>(p & 15) * 64 + c * 8;
        ao_cp16(smem_u32(dK + t * kAoKS + c * 8), src, ok);
        ao_cp16(smem_u32(dV + t * kAoKS + c * 8), ok ? src + Hkv * 16 * 64 : layer_base, ok);
      }
    };
    const int pre_hi = max(w_lo, min(stable, w_hi));
    for (int j = 0; j < kAoBuf && j < nsub_all; ++j) issue(j, w_lo, pre_hi, pre_hi);   // rows written before the step
    pdl_wait();
    for (int j = 0; j < kAoBuf; ++j) {                // the step's own rows, then one group per sub-tile
      if (j < nsub_all) issue(j, pre_hi, INT_MAX, w_hi);
      ao_commit();
    }
    if (at < 128) pf = first_pair_ops(a, rank, sp, NT, first_tile, at);
    {  // queries of the group's rows on this KV head -> bf16, row positions
      const int qv = at >> 4, c4 = at & 15;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (qv < nqv)
        v = __ldcg(reinterpret_cast<const float4*>(a.attn_q + (static_cast<size_t>(qv / G) * a.n_heads + kvh * G + qv % G) * 64) + c4);
      *reinterpret_cast<uint2*>(sQ + qv * kAoKS + c4 * 4) = make_uint2(ao_pack(v.x, v.y), ao_pack(v.z, v.w));
      if (at < 16) sPos[at] = at < nqv ? __ldcg(a.row_pos + at / G) : -1;
    }
    named_bar_attn();
    int pmax = -1;
#pragma unroll
    for (int i = 0; i < 16; ++i) pmax = max(pmax, sPos[i]);
    if (at == 0 && pmax + 1 > ctx_hi && a.err) atomicOr(a.err, static_cast<unsigned>(ERR_RANGE));
    const int hi = min(pmax + 1, w_hi);
    const int nsub = hi > w_lo ? (hi - w_lo + kAoSub - 1) / kAoSub : 0;
    const int pa = sPos[g8], pb = sPos[g8 + 8];
    uint32_t qa[4][4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const bf16* q0 = sQ + g8 * kAoKS + kk * 16 + 2 * t4;
      qa[kk][0] = ao_ld_u32(q0);
      qa[kk][1] = ao_ld_u32(q0 + 8 * kAoKS);
      qa[kk][2] = ao_ld_u32(q0 + 8);
      qa[kk][3] = ao_ld_u32(q0 + 8 * kAoKS + 8);
    }
    float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;
    float acc[8][4];
#pragma unroll
    for (int dt = 0; dt < 8; ++dt) acc[dt][0] = acc[dt][1] = acc[dt][2] = acc[dt][3] = 0.f;
    for (int j = 0; j < nsub; ++j) {
      ao_wait<kAoBuf - 1>();
      __syncwarp();
      const bf16* sK = reinterpret_cast<const bf16*>(wkv + (j % kAoBuf) * 2 * kAoSub * kAoKS * 2);
      const bf16* sV = sK + kAoSub * kAoKS;
      float sc[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const bf16* kp = sK + (nt * 8 + g8) * kAoKS + kk * 16 + 2 * t4;
          ao_mma(c, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], ao_ld_u32(kp), ao_ld_u32(kp + 8));
        }
        const int pc = w_lo + j * kAoSub + nt * 8 + 2 * t4;
        sc[nt][0] = pc <= pa ? c[0] * 0.125f : -INFINITY;
        sc[nt][1] = pc + 1 <= pa ? c[1] * 0.125f : -INFINITY;
        sc[nt][2] = pc <= pb ? c[2] * 0.125f : -INFINITY;
        sc[nt][3] = pc + 1 <= pb ? c[3] * 0.125f : -INFINITY;
      }
      float mx_a = fmaxf(fmaxf(sc[0][0], sc[0][1]), fmaxf(sc[1][0], sc[1][1]));
      float mx_b = fmaxf(fmaxf(sc[0][2], sc[0][3]), fmaxf(sc[1][2], sc[1][3]));
      mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
      mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
      mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
      mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
      const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
      const float mu_a = mn_a == -INFINITY ? 0.f : mn_a, mu_b = mn_b == -INFINITY ? 0.f : mn_b;
      const float cr_a = __expf(m_a - mu_a), cr_b = __expf(m_b - mu_b);
      m_a = mn_a;
      m_b = mn_b;
      uint32_t pk[4];
      float ps_a = 0.f, ps_b = 0.f;
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        const __nv_bfloat162 ha = __floats2bfloat162_rn(__expf(sc[nt][0] - mu_a), __expf(sc[nt][1] - mu_a));
        const __nv_bfloat162 hb = __floats2bfloat162_rn(__expf(sc[nt][2] - mu_b), __expf(sc[nt][3] - mu_b));
        ps_a += __low2float(ha) + __high2float(ha);
        ps_b += __low2float(hb) + __high2float(hb);
        pk[2 * nt] = *reinterpret_cast<const uint32_t*>(&ha);
        pk[2 * nt + 1] = *reinterpret_cast<const uint32_t*>(&hb);
      }
      l_a = l_a * cr_a + ps_a;
      l_b = l_b * cr_b + ps_b;
      const int vrow = (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
      for (int dt = 0; dt < 8; ++dt) {
        acc[dt][0] *= cr_a; acc[dt][1] *= cr_a;
        acc[dt][2] *= cr_b; acc[dt][3] *= cr_b;
        uint32_t v0, v1;
        ao_ldsm_x2_t(smem_u32(sV + vrow * kAoKS + dt * 8), v0, v1);
        ao_mma(acc[dt], pk[0], pk[1], pk[2], pk[3], v0, v1);
      }
      __syncwarp();                                    // every lane is done with this slot
      if (j + kAoBuf < nsub) issue(j + kAoBuf, w_lo, INT_MAX, w_hi);
      ao_commit();
    }
    ao_wait<0>();
    __syncwarp();
    l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
    l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
    l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
    l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);
    // this warp's partial over its positions, over its own K/V buffers
    float* pacc = reinterpret_cast<float*>(wkv);        // [16 rows][kAoAS]
#pragma unroll
    for (int dt = 0; dt < 8; ++dt) {
      *reinterpret_cast<float2*>(pacc + g8 * kAoAS + dt * 8 + 2 * t4) = make_float2(acc[dt][0], acc[dt][1]);
      *reinterpret_cast<float2*>(pacc + (g8 + 8) * kAoAS + dt * 8 + 2 * t4) = make_float2(acc[dt][2], acc[dt][3]);
    }
    if (t4 == 0) {
      sML[(aw * 16 + g8) * 2] = m_a;
      sML[(aw * 16 + g8) * 2 + 1] = l_a;
      sML[(aw * 16 + g8 + 8) * 2] = m_b;
      sML[(aw * 16 + g8 + 8) * 2 + 1] = l_b;
    }
    named_bar_attn();
    // merge over the 8 warps (in warp order) -> the token operand: stage s holds head s of the KV
    // head, token row t at byte t * 128 of the stage's operand, 16-byte chunk ch at (ch ^ (t & 7))
    for (int e = at; e < NT * S * 8; e += 256) {
      const int ch = e & 7, sgi = (e >> 3) % S, t = (e >> 3) / S;
      uint4 pkd = make_uint4(0u, 0u, 0u, 0u);
      if (t < M) {
        const int qv = t * G + sgi;
        float mw[8], M_ = -INFINITY;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
          mw[w] = sML[(w * 16 + qv) * 2];
          M_ = fmaxf(M_, mw[w]);
        }
        float L = 0.f, o[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int w = 0; w < 8; ++w) {
          const float ww = __expf(mw[w] - M_);
          L += sML[(w * 16 + qv) * 2 + 1] * ww;
          const float* src = reinterpret_cast<const float*>(sKV + static_cast<size_t>(w) * kAoWarpBytes) + qv * kAoAS + ch * 8;
#pragma unroll
          for (int d = 0; d < 8; ++d) o[d] = fmaf(ww, src[d], o[d]);
        }
        const float inv = L > 0.f ? 1.f / L : 0.f;
        pkd = make_uint4(ao_pack(o[0] * inv, o[1] * inv), ao_pack(o[2] * inv, o[3] * inv), ao_pack(o[4] * inv, o[5] * inv),
                         ao_pack(o[6] * inv, o[7] * inv));
      }
      *reinterpret_cast<uint4*>(smem + static_cast<size_t>(sgi) * stage_bytes + a_bytes + t * 128 + ((ch ^ (t & 7)) << 4)) = pkd;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // the operand is read by the tensor cores
    named_bar_attn();
    if (at == 0)
      for (int j = 0; j < S; ++j) mbar_arrive(full0 + 8 * j);
    if (warp < 6)                                       // warps 2-5: the split-K epilogue
      splitk_epilogue(a, SplitK{smem, recv, rs, flags, tfull0, rbar, tmem, rank, sp, npmax, NT, first_tile}, warp, lane, pf);
  }
  if (warp < 2 || warp >= 6) {                          // everyone but the epilogue takes its half of the cluster barrier
    __syncwarp();
    cluster_wait();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 32);
}

// ------------------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

bool make_map(CUtensorMap* map, const void* base, int rows, int K, int ld, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Weight maps never change: encode each (pointer, shape) once.
bool weight_map(CUtensorMap* out, const void* w, int rows, int K, int box_rows) {
  struct Key {
    const void* p;
    int rows, K, box;
    bool operator==(const Key& o) const { return p == o.p && rows == o.rows && K == o.K && box == o.box; }
  };
  struct H {
    size_t operator()(const Key& k) const {
      return std::hash<const void*>()(k.p) ^ (static_cast<size_t>(k.rows) << 20) ^ (static_cast<size_t>(k.K) << 4) ^
             static_cast<size_t>(k.box);
    }
  };
  static std::unordered_map<Key, CUtensorMap, H> cache;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  const Key key{w, rows, K, box_rows};
  auto it = cache.find(key);
  if (it != cache.end()) { *out = it->second; return true; }
  if (!make_map(out, w, rows, K, K, box_rows)) return false;
  cache.emplace(key, *out);
  return true;
}

int sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

constexpr int kSmemBudget = 227 * 1024;
constexpr int kSmemShared = 110 * 1024;

// Registers a thread of the most demanding instantiation of gemm_tc_kernel uses (0 if unknown).
int gemm_tc_max_regs() {
  static const int regs = [] {
    int r = 0;
    auto take = [&](const void* f) {
      cudaFuncAttributes fa{};
      if (cudaFuncGetAttributes(&fa, f) == cudaSuccess) r = std::max(r, fa.numRegs);
      else r = -1000;
    };
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgs, 1>));
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgs, 2>));
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgsE<EPI_STORE>, 0>));
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgsE<EPI_ADD>, 0>));
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgsE<EPI_SWIGLU>, 0>));
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgsE<EPI_QKV>, 0>));
    take(reinterpret_cast<const void*>(gemm_tc_kernel<TcArgsE<EPI_SILU>, 0>));
    cudaGetLastError();
    return r;
  }();
  return regs;
}

// Stand-in for gemm_tc_kernel in residency queries: the same block size and launch bounds, no
// tensor memory. The occupancy calculator reports one CTA per SM for gemm_tc_kernel at any shared
// memory size (measured: 152 clusters of 1, 76 of 2, ... even at 60 KB), while the hardware places
// two of its CTAs on an SM whenever their shared memory fits (per-CTA %smid traces of its launches);
// for this kernel the calculator's answers match a measured first wave at every size. Never launched.
__global__ void __launch_bounds__(kThreads, 2) residency_proxy_kernel() {}

// Clusters of `size` CTAs with `smem` bytes of dynamic shared memory each that the device holds at
// once. Clusters must fit whole into a GPC, so this is less than SMs x (CTAs per SM) / size: at two
// CTAs per SM, 97 clusters of 3 or 36 of 8; at one, 46 of 3 or 15 of 7 on a 152-SM GB300. The
// registers of gemm_tc_kernel must allow two CTAs per SM for the two-per-SM figures to hold; if they
// do not, one CTA per SM is assumed. Cached per (size, smem).
int max_active_clusters(int size, int smem) {
  static std::mutex mu;
  static std::unordered_map<long long, int> cache;
  const long long key = (static_cast<long long>(size) << 32) | static_cast<unsigned>(smem);
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  // registers are allocated per warp in units of 256
  const int regs = gemm_tc_max_regs();
  const bool two_fit = regs > 0 && 2 * (kThreads / 32) * ((regs * 32 + 255) / 256 * 256) <= 65536;
  // one CTA per SM when the registers say so: pad the shared memory beyond half an SM
  const int q_smem = (!two_fit && smem <= kSmemShared) ? kSmemShared + 4096 : smem;
  int n = 0;
  if (cudaFuncSetAttribute(residency_proxy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget) ==
      cudaSuccess) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(size));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = static_cast<size_t>(q_smem);
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = static_cast<unsigned>(size);
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, residency_proxy_kernel, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();
  cache.emplace(key, n);
  return n;
}

// Launch shape of a grid of `tiles` weight tiles x token tiles: split factor sp (CTAs per tile, one
// cluster), ring stages, dynamic shared memory and grid. Two CTAs share an SM when the ring (at
// least 3 stages) and the split-K receive buffer fit in half its shared memory: more weight bytes in
// flight per SM, and room for the next kernel's CTAs to start early. With fewer tiles than resident
// CTAs the K range is split, aiming at 2 CTAs per SM (two-per-SM plans) or one (one-per-SM plans),
// never past one wave. Of the two, the plan with more CTAs streaming at once wins (ties: two per SM).
struct TcPlan {
  int sp = 0, stages = 0, smem = 0, grid = 0;
};
TcPlan plan_tc(int tiles, int NT, int KB) {
  const int sms = sm_count();
  const int stage_bytes = (kWRows + NT) * kBK * 2;
  auto fixed_of = [&](int sp) {
    const int recv = sp > 1 ? sp * ((64 + sp - 1) / sp) * 2 * NT * 4 : 0;   // split-K receive buffer
    return 1024 + recv + kWRows * kXS * 4 + 64 + kMaxNT * 4 + 8 * (2 * 16 + 6);
  };
  TcPlan best;
  int best_active = 0;
  for (int occ = 2; occ >= 1; --occ) {
    const int budget = occ == 2 ? kSmemShared : kSmemBudget;
    // Wide token tiles (NT > 128) take two CTAs per SM only as one whole tile per CTA: a single
    // accumulator (at most 256 TMEM columns, so two CTAs fit), and a two-stage ring is accepted.
    const bool wide = NT > 128;
    if (occ == 2 && wide && tiles > 2 * sms) continue;
    const int min_stages = occ == 2 && !wide ? 3 : 2;
    int sp = 1;
    if (tiles < sms * occ) {                             // split-K tiles keep one NT-column accumulator
      sp = ((occ == 2 ? 2 * sms : sms) + tiles / 2) / tiles;
      sp = std::max(1, std::min(sp, std::min(8, KB)));
      while (sp > 1 && tiles * sp > sms * occ) --sp;
    }
    for (; sp >= 1; --sp) {
      const int S = std::min(8, (budget - fixed_of(sp)) / stage_bytes);
      if (S < min_stages) continue;
      TcPlan pl;
      pl.sp = sp;
      pl.stages = S;
      pl.smem = fixed_of(sp) + S * stage_bytes;
      // every tile's cluster must be resident in the one wave (a cluster left over would run after
      // the others and double the launch's time)
      if (sp > 1 && max_active_clusters(sp, pl.smem) < tiles) continue;
      pl.grid = sp > 1 ? tiles * sp : std::min(tiles, occ * sms);
      const int active = std::min(pl.grid, occ * sms);
      if (active > best_active) {
        best = pl;
        best_active = active;
      }
      break;
    }
  }
  return best;
}

int n_out_rows(const GemmArgs& g) {
  int N = 0;
  for (int s = 0; s < g.nseg; ++s) N += g.seg[s].rows;
  return N;
}

}  // namespace

bool encode_weight_map(void* map, const void* w, int rows, int K, int box_rows) {
  return make_map(static_cast<CUtensorMap*>(map), w, rows, K, K, box_rows);
}

int sm_count_cached() { return sm_count(); }

int gemm_norm_parts(const GemmArgs& g) {
  if (g.attn_q) return (g.seg[0].rows / kWRows) * g.n_kv_heads;   // fused attention: sp = H_kv
  const int NT = gemm_tc_token_tile(g.M);
  const int n_wtiles = n_out_rows(g) / kWRows;
  const int tiles = n_wtiles * ((g.M + NT - 1) / NT);
  return n_wtiles * std::max(1, plan_tc(tiles, NT, g.K / kBK).sp);
}

int gemm_tc_token_tile(int M) {
  int nt = ((M + 15) / 16) * 16;
  return nt > 256 ? 256 : (nt < 16 ? 16 : nt);
}


bool gemm_tc_supported(const GemmArgs& g) {
  if (g.K % kBK != 0 || g.K < kBK || g.M < 1 || g.ldx % 8 != 0) return false;
  if (reinterpret_cast<uintptr_t>(g.x) & 15) return false;
  if (g.epi == EPI_QKV && (g.head_dim != 64 && g.head_dim != 128)) return false;
  if (g.norm_out && (g.epi != EPI_ADD || !g.norm_gamma || !g.norm_ssq_out)) return false;
  if (g.tap_mask && (!g.norm_out || !g.tap)) return false;
  if (g.norm_ssq_in && (g.epi == EPI_ADD || g.norm_parts < 1 || g.norm_d < 1)) return false;
  if (g.epi == EPI_SWIGLU) return g.nseg == 2 && g.seg[0].rows == g.seg[1].rows && g.seg[0].rows % 64 == 0;
  for (int s = 0; s < g.nseg; ++s)
    if (g.seg[s].rows % kWRows != 0) return false;
  return true;
}

// Shared memory of the fused attention kernel for S k-blocks per rank and token tile NT.
size_t gemm_attn_smem(int S, int NT, int sp) {
  const size_t stage_bytes = static_cast<size_t>(kWRows + NT) * kBK * 2;
  const size_t recv = static_cast<size_t>(sp) * ((64 + sp - 1) / sp) * 2 * NT * 4;
  return 1024 + S * stage_bytes + recv + 8 * (2 * S + 6) + 16 * 4 + 16 * 4 + kAoAttnBytes;
}

bool gemm_attn_supported(const GemmArgs& g) {
  if (!g.attn_q || !g.attn_seq || !g.attn_pre_len || !g.kv_pool || !g.kv_table || !g.row_pos) return false;
  if (g.epi != EPI_ADD || g.nseg != 1 || g.norm_ssq_in || g.head_dim != 64) return false;
  if (g.n_kv_heads < 2 || g.n_kv_heads > 8 || g.n_heads % g.n_kv_heads || g.K != g.n_heads * 64) return false;
  if (g.norm_out && (!g.norm_gamma || !g.norm_ssq_out)) return false;
  if (g.tap_mask && (!g.norm_out || !g.tap)) return false;
  const int G = g.n_heads / g.n_kv_heads;
  if (g.M < 1 || g.M * G > 16 || g.seg[0].rows % kWRows != 0) return false;
  if (g.kv_bt_stride < 1 || g.kv_bt_stride * 16 > 8 * kAoMaxBlk * 16) return false;   // context <= 4096
  const int tiles = g.seg[0].rows / kWRows;
  if (tiles * g.n_kv_heads > sm_count()) return false;   // one CTA per SM, one wave
  return gemm_attn_smem(G, gemm_tc_token_tile(g.M), g.n_kv_heads) <= static_cast<size_t>(kSmemBudget);
}

cudaError_t gemm_attn(const GemmArgs& g, unsigned* err, cudaStream_t st) {
  TcArgs a{};
  a.nseg = 1;
  a.seg_rows[0] = g.seg[0].rows;
  if (!weight_map(&a.mapA[0], g.seg[0].w, g.seg[0].rows, g.K, kWRows)) return cudaErrorInvalidValue;
  a.NT = gemm_tc_token_tile(g.M);
  a.M = g.M; a.K = g.K; a.KB = g.K / kBK;
  a.n_wtiles = g.seg[0].rows / kWRows;
  a.n_ttiles = 1;
  a.tiles = a.n_wtiles;
  a.epi = EPI_ADD; a.out = g.out; a.ldo = g.ldo;
  a.bias = g.bias; a.ld_bias = g.ld_bias; a.row_seq = g.row_seq;
  a.err = err;
  a.kv_pool = static_cast<bf16*>(g.kv_pool); a.kv_table = g.kv_table;
  a.kv_bt_stride = g.kv_bt_stride; a.kv_n_blocks = g.kv_n_blocks; a.n_heads = g.n_heads;
  a.n_kv_heads = g.n_kv_heads; a.head_dim = 64; a.layer = g.layer; a.row_pos = g.row_pos;
  a.norm_gamma = static_cast<const bf16*>(g.norm_gamma); a.norm_out = static_cast<bf16*>(g.norm_out);
  a.norm_ssq_out = g.norm_ssq_out; a.tap = g.tap; a.tap_row = g.tap_row; a.tap_mask = g.tap_mask;
  a.ld_ssq = g.ld_ssq;
  a.attn_q = g.attn_q; a.attn_seq = g.attn_seq; a.attn_pre_len = g.attn_pre_len;
  a.attn_pre_stable = g.attn_pre_stable; a.attn_pre_fresh = g.attn_pre_fresh;
  a.sp = g.n_kv_heads;
  a.stages = g.n_heads / g.n_kv_heads;
  const size_t smem = gemm_attn_smem(a.stages, a.NT, a.sp);
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(gemm_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  return launch_pdl_cluster(gemm_attn_kernel, dim3(static_cast<unsigned>(a.tiles * a.sp)), dim3(kAoThreads), smem, st,
                            a.sp, a);
}

namespace {
// One launch of the instantiation for argument type A (its shared-memory opt-in set once).
template <class A, int SPLIT>
cudaError_t launch_tc(const TcArgs& a, const TcPlan& pl, cudaStream_t st) {
  static const cudaError_t configured =
      cudaFuncSetAttribute(gemm_tc_kernel<A, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget);
  if (configured != cudaSuccess) return configured;
  A ae;
  static_cast<TcArgs&>(ae) = a;
  return launch_pdl_cluster(gemm_tc_kernel<A, SPLIT>, dim3(static_cast<unsigned>(pl.grid)), dim3(kThreads),
                            static_cast<size_t>(pl.smem), st, pl.sp, ae);
}
}  // namespace

cudaError_t gemm_tc(const GemmArgs& g, unsigned* err, cudaStream_t st) {
  if (g.attn_q) return gemm_attn(g, err, st);
  TcArgs a{};  // built on the host; passed by value as the kernel parameter
  a.nseg = g.nseg;
  a.swiglu = (g.epi == EPI_SWIGLU) ? 1 : 0;
  int N = 0;
  for (int s = 0; s < g.nseg; ++s) {
    a.seg_rows[s] = g.seg[s].rows;
    N += g.seg[s].rows;
    if (!weight_map(&a.mapA[s], g.seg[s].w, g.seg[s].rows, g.K, a.swiglu ? 64 : kWRows))
      return cudaErrorInvalidValue;
  }
  a.NT = gemm_tc_token_tile(g.M);
  if (!make_map(&a.mapB, g.x, g.M, g.K, g.ldx, a.NT)) return cudaErrorInvalidValue;
  a.M = g.M; a.K = g.K; a.KB = g.K / kBK;
  a.n_wtiles = a.swiglu ? g.seg[0].rows / 64 : N / kWRows;
  a.n_ttiles = (g.M + a.NT - 1) / a.NT;
  a.tiles = a.n_wtiles * a.n_ttiles;
  a.epi = g.epi; a.out = g.out; a.ldo = g.ldo; a.out_bf = static_cast<bf16*>(g.out_bf); a.ldh = g.ldh;
  a.bias = g.bias; a.ld_bias = g.ld_bias; a.row_seq = g.row_seq;
  a.err = err;
  a.stamp = g.stamp;
  a.q_out = g.q_out; a.kv_pool = static_cast<bf16*>(g.kv_pool); a.kv_table = g.kv_table;
  a.kv_bt_stride = g.kv_bt_stride; a.kv_n_blocks = g.kv_n_blocks; a.n_heads = g.n_heads;
  a.n_kv_heads = g.n_kv_heads; a.head_dim = g.head_dim; a.layer = g.layer; a.rope_cs = g.rope_cs;
  a.row_pos = g.row_pos; a.row_valid = g.row_valid;
  a.norm_gamma = static_cast<const bf16*>(g.norm_gamma); a.norm_out = static_cast<bf16*>(g.norm_out);
  a.norm_ssq_out = g.norm_ssq_out; a.tap = g.tap; a.tap_row = g.tap_row; a.tap_mask = g.tap_mask;
  a.norm_ssq_in = g.norm_ssq_in; a.norm_parts = g.norm_parts; a.norm_d = g.norm_d; a.norm_eps = g.norm_eps;
  a.ld_ssq = g.ld_ssq;
  const TcPlan pl = plan_tc(a.tiles, a.NT, a.KB);
  if (pl.sp < 1) return cudaErrorInvalidValue;
  const int sp = pl.sp;
  a.sp = sp;
  a.stages = pl.stages;
  // Narrow token tiles (up to 16 columns: batch-1 decode) share one kernel whatever the epilogue:
  // their launches are short, and one body of code stays warm in the instruction caches across
  // a layer's projections (per-epilogue kernels made the 1B drafter step 4% slower). Wider tiles,
  // whose owner passes run many outputs per thread, take the kernel of their own epilogue.
  if (a.NT <= 16) return sp > 1 ? launch_tc<TcArgs, 1>(a, pl, st) : launch_tc<TcArgs, 2>(a, pl, st);
  switch (a.epi) {
    case EPI_STORE: return launch_tc<TcArgsE<EPI_STORE>, 0>(a, pl, st);
    case EPI_ADD: return launch_tc<TcArgsE<EPI_ADD>, 0>(a, pl, st);
    case EPI_SWIGLU: return launch_tc<TcArgsE<EPI_SWIGLU>, 0>(a, pl, st);
    case EPI_QKV: return launch_tc<TcArgsE<EPI_QKV>, 0>(a, pl, st);
    case EPI_SILU: return launch_tc<TcArgsE<EPI_SILU>, 0>(a, pl, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace sd2
