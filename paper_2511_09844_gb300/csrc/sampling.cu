// Speculative acceptance (Sec. 3.1; Leviathan et al. 2023) and token sampling over the
// vocabulary.
//
// Decisions are integers (token ids, accept/reject), so every floating-point step that feeds one
// is a correctly rounded fp32 operation in a fixed order (common.cuh: exp_cw, log_at), and every
// reduction across threads and CTAs is exact: maxima and arg-maxima through atomicMax on
// order-preserving packed keys (ties to the lowest index), the softmax normaliser through 64-bit
// integer sums of floor(e * 2^45). The outcome therefore does not depend on how the vocabulary
// is split across CTAs.
//
//   p = softmax(z / T):  s = z * fl(1/T), m = max s, e = exp(s - m), S = fl(sum floor(e 2^45)) 2^-45,
//                        p = e / S
//   accept draft i  iff  u_i * q_i(x_i) <= p_{i-1}(x_i)              (u_i from Philox)
//   replacement         argmax_v max(0, p_j - q_{j+1})_v / E_v, E_v = -ln u_v; if that residual is 0
//                        everywhere, argmax_v (s_v - ln E_v) on row j
//   bonus / draft       argmax_v (s_v - ln E_v)   (exponential race in log form)
//   T = 0               accept iff x_i = argmax z_{i-1}; emit argmax of the row
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace sd2 {
namespace {

constexpr int kThreads = 256;
constexpr int kPerCta = kThreads * 4 * 8;   // most vocabulary entries per CTA (8 passes of 4 per thread)
constexpr int kStatsPerCta = kThreads * 8 * 8;   // the row-statistics passes: at most 8 passes of 8
enum { MODE_NONE = 0, MODE_DONE = 1, MODE_RESIDUAL = 2, MODE_BONUS = 3 };

// Vocabulary entries per CTA for `rows` rows: enough CTAs per row to fill the GPU about twice over,
// in whole passes of `gran` entries per thread, at most max_span (few rows: more, shorter CTAs; a
// large batch keeps long ones). Every decision is independent of how the vocabulary is split.
int vocab_span(int V, int rows, int gran, int max_span) {
  const int pass = kThreads * gran;
  const int want = std::max(1, (2 * sm_count_cached() + rows - 1) / std::max(1, rows));
  const int span = (((V + want - 1) / want + pass - 1) / pass) * pass;
  return std::min(max_span, std::max(pass, span));
}

template <typename T>
__device__ __forceinline__ void load4(const T* row, int v, float z[4]);
template <>
__device__ __forceinline__ void load4<float>(const float* row, int v, float z[4]) {
  const float4 t = *reinterpret_cast<const float4*>(row + v);
  z[0] = t.x; z[1] = t.y; z[2] = t.z; z[3] = t.w;
}
template <>
__device__ __forceinline__ void load4<bf16>(const bf16* row, int v, float z[4]) {
  const uint2 t = *reinterpret_cast<const uint2*>(row + v);
  z[0] = bf_lo(t.x); z[1] = bf_hi(t.x); z[2] = bf_lo(t.y); z[3] = bf_hi(t.y);
}
// 8 consecutive entries from v (n < 8 of them at the row's end; rows start 16-byte (f32) or 8-byte
// (bf16) aligned)
template <typename T>
__device__ __forceinline__ void load8(const T* row, int v, int n, float z[8]);
template <>
__device__ __forceinline__ void load8<float>(const float* row, int v, int n, float z[8]) {
  if (n >= 8) {
    const float4 a = *reinterpret_cast<const float4*>(row + v), b = *reinterpret_cast<const float4*>(row + v + 4);
    z[0] = a.x; z[1] = a.y; z[2] = a.z; z[3] = a.w; z[4] = b.x; z[5] = b.y; z[6] = b.z; z[7] = b.w;
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) z[j] = j < n ? row[v + j] : 0.f;
  }
}
template <>
__device__ __forceinline__ void load8<bf16>(const bf16* row, int v, int n, float z[8]) {
  if (n >= 8) {    // rows are 8-byte aligned (V % 4 == 0): two 8-byte loads
    const uint2 t = *reinterpret_cast<const uint2*>(row + v), u = *reinterpret_cast<const uint2*>(row + v + 4);
    z[0] = bf_lo(t.x); z[1] = bf_hi(t.x); z[2] = bf_lo(t.y); z[3] = bf_hi(t.y);
    z[4] = bf_lo(u.x); z[5] = bf_hi(u.x); z[6] = bf_lo(u.y); z[7] = bf_hi(u.y);
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) z[j] = j < n ? bf2f(row[v + j]) : 0.f;
  }
}
template <typename T>
__device__ __forceinline__ float load1(const T* row, int v);
template <>
__device__ __forceinline__ float load1<float>(const float* row, int v) { return row[v]; }
template <>
__device__ __forceinline__ float load1<bf16>(const bf16* row, int v) { return bf2f(row[v]); }

__device__ __forceinline__ float inv_temp(float t) { return __fdiv_rn(1.0f, t); }

__device__ __forceinline__ unsigned long long block_max_u64(unsigned long long v, unsigned long long* red) {
  v = warp_max_u64(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  v = (l < (int)(blockDim.x >> 5)) ? red[l] : 0ull;
  return warp_max_u64(v);
}
__device__ __forceinline__ unsigned long long block_sum_u64(unsigned long long v, unsigned long long* red) {
  v = warp_sum_u64(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  v = (l < (int)(blockDim.x >> 5)) ? red[l] : 0ull;
  return warp_sum_u64(v);
}

struct RowRef {
  int b;
  bool is_draft;
  size_t offset;  // element offset of the row
};
// Row r of the stats table: target rows b*(k+1)+i first, then draft rows b*k+i.
__device__ __forceinline__ RowRef row_ref(int r, int B, int k, int V) {
  RowRef rr;
  const int nt = B * (k + 1);
  if (r < nt) {
    rr.b = r / (k + 1); rr.is_draft = false; rr.offset = static_cast<size_t>(r) * V;
  } else {
    rr.b = (r - nt) / k; rr.is_draft = true; rr.offset = static_cast<size_t>(r - nt) * V;
  }
  return rr;
}

__device__ __forceinline__ unsigned step_value(const int* step_ptr, unsigned step) {
  return step_ptr ? static_cast<unsigned>(*step_ptr) : step;
}
__device__ __forceinline__ unsigned long long seed_value(const Seed& s) { return s.ptr ? *s.ptr : s.value; }

// Pass 1: packed (max, argmax) of s = z/T (or z at T = 0) per row.
template <typename T>
__global__ void __launch_bounds__(kThreads) rowmax_kernel(const T* target, const T* draft, int B, int k, int V,
                                                          const float* temp, const int* stopped,
                                                          unsigned long long* rowkey, unsigned long long* rowsum,
                                                          unsigned* err, int span) {
  pdl_trigger();
  pdl_wait();
  __shared__ unsigned long long red[32];
  // the normaliser pass adds into rowsum; it runs after this grid has completed
  if (blockIdx.y == 0 && threadIdx.x == 0) rowsum[blockIdx.x] = 0ull;
  const RowRef rr = row_ref(blockIdx.x, B, k, V);
  if (stopped && stopped[rr.b]) return;
  const float t = temp[rr.b];
  const bool greedy = !(t > 0.f);
  if (greedy && rr.is_draft) return;
  const float invT = greedy ? 1.f : inv_temp(t);
  const T* row = (rr.is_draft ? draft : target) + rr.offset;
  const int lo = blockIdx.y * span, hi = min(V, lo + span);
  // this thread's (max, first index of it) in 32 bits: its entries come in increasing index order,
  // so a strictly greater value is the only update (+0 and -0 compare equal, as the packed key
  // folds them); packed once for the exact cross-thread maximum
  // Each group of 8 is reduced with fmaxf first; only a group that beats the running maximum is
  // searched for the first index of its maximum. Non-finite entries show as a NaN in sum(z - z).
  float best_s = -INFINITY;
  int best_i = -1;
  float nf = 0.f;
#pragma unroll 2
  for (int v = lo + threadIdx.x * 8; v < hi; v += kThreads * 8) {
    float z[8];
    const int n = min(8, hi - v);
    load8<T>(row, v, n, z);
    float s[8];
    if (n == 8) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        nf += __fsub_rn(z[j], z[j]);
        s[j] = greedy ? z[j] : __fmul_rn(z[j], invT);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        nf += j < n ? __fsub_rn(z[j], z[j]) : 0.f;
        s[j] = j < n ? (greedy ? z[j] : __fmul_rn(z[j], invT)) : -INFINITY;
      }
    }
    const float g = fmaxf(fmaxf(fmaxf(s[0], s[1]), fmaxf(s[2], s[3])), fmaxf(fmaxf(s[4], s[5]), fmaxf(s[6], s[7])));
    if (g > best_s || best_i < 0) {
      int jj = 7;
#pragma unroll
      for (int j = 7; j >= 0; --j) jj = (j < n && s[j] == g) ? j : jj;
      if (g > best_s || best_i < 0) { best_s = g; best_i = v + jj; }
    }
  }
  const bool bad = !(nf == 0.f);
  unsigned long long best = best_i < 0 ? 0ull : pack_key(best_s, static_cast<uint32_t>(best_i));
  best = block_max_u64(best, red);
  if (threadIdx.x == 0) atomicMax(&rowkey[blockIdx.x], best);
  if (bad) atomicOr(err, static_cast<unsigned>(ERR_NONFINITE));
}

// Pass 2: exact fixed-point normaliser sum floor(exp(s - m) * 2^45) per sampled row.
template <typename T>
__global__ void __launch_bounds__(kThreads) rowsum_kernel(const T* target, const T* draft, int B, int k, int V,
                                                          const float* temp, const int* stopped,
                                                          const unsigned long long* rowkey,
                                                          unsigned long long* rowsum, int span) {
  pdl_trigger();
  pdl_wait();
  __shared__ unsigned long long red[32];
  const RowRef rr = row_ref(blockIdx.x, B, k, V);
  if (stopped && stopped[rr.b]) return;
  const float t = temp[rr.b];
  if (!(t > 0.f)) return;
  const float invT = inv_temp(t);
  const float m = packed_key(rowkey[blockIdx.x]);
  const T* row = (rr.is_draft ? draft : target) + rr.offset;
  const int lo = blockIdx.y * span, hi = min(V, lo + span);
  uint32_t acc_hi = 0, acc_lo = 0;        // at most 64 entries per thread: no overflow
#pragma unroll 2
  for (int v = lo + threadIdx.x * 8; v < hi; v += kThreads * 8) {
    float z[8];
    const int n = min(8, hi - v);
    load8<T>(row, v, n, z);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < n) {
        uint32_t ph, pl;
        fixed45_parts(exp_cw(__fsub_rn(__fmul_rn(z[j], invT), m)), ph, pl);
        acc_hi += ph;
        acc_lo += pl;
      }
  }
  unsigned long long acc = (static_cast<unsigned long long>(acc_hi) << 23) + acc_lo;
  acc = block_sum_u64(acc, red);
  if (threadIdx.x == 0 && acc) atomicAdd(&rowsum[blockIdx.x], acc);
}

struct RowDist {  // what p(x) needs for one row
  float m, S;
};
__device__ __forceinline__ RowDist row_dist(const unsigned long long* rowkey, const unsigned long long* rowsum, int r) {
  RowDist d;
  d.m = packed_key(rowkey[r]);
  d.S = __fmul_rn(__ull2float_rn(rowsum[r]), 0x1p-45f);
  return d;
}
__device__ __forceinline__ float prob(float z, float invT, RowDist d) {
  return __fdiv_rn(exp_cw(__fsub_rn(__fmul_rn(z, invT), d.m)), d.S);
}

// Sequential decisions of one block per sequence (one thread per sequence).
template <typename T>
__global__ void decide_kernel(const T* target, const T* draft, const int* xhat, const float* temp, int B, int k, int V,
                              Seed seed_arg, const int* step_ptr, unsigned step, const int* stopped,
                              const unsigned long long* rowkey, const unsigned long long* rowsum, int* tokens, int* n,
                              AcceptScratch s) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  s.slot[2 * b] = 0ull;
  s.slot[2 * b + 1] = 0ull;
  s.counter[b] = 0;
  int* out = tokens + static_cast<size_t>(b) * (k + 1);
  if (stopped && stopped[b]) {
    n[b] = 0;
    s.jmode[2 * b] = 0;
    s.jmode[2 * b + 1] = MODE_NONE;
    return;
  }
  const int* xb = xhat + static_cast<size_t>(b) * k;
  const float t = temp[b];
  const int nt = B * (k + 1);
  if (!(t > 0.f)) {
    int j = k;
    for (int i = 1; i <= k; ++i) {
      if (xb[i - 1] != static_cast<int>(packed_index(rowkey[b * (k + 1) + i - 1]))) { j = i - 1; break; }
    }
    for (int i = 0; i < j; ++i) out[i] = xb[i];
    out[j] = static_cast<int>(packed_index(rowkey[b * (k + 1) + j]));
    n[b] = j + 1;
    s.jmode[2 * b] = j;
    s.jmode[2 * b + 1] = MODE_DONE;
    return;
  }
  const float invT = inv_temp(t);
  const unsigned stp = step_value(step_ptr, step);
  const unsigned long long seed = seed_value(seed_arg);
  const uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
  int j = k;
  for (int i = 1; i <= k; ++i) {
    const int x = min(max(xb[i - 1], 0), V - 1);
    const int rt = b * (k + 1) + i - 1, rd = nt + b * k + i - 1;
    const float p = prob(load1<T>(target + static_cast<size_t>(rt) * V, x), invT, row_dist(rowkey, rowsum, rt));
    const float q = prob(load1<T>(draft + static_cast<size_t>(rd - nt) * V, x), invT, row_dist(rowkey, rowsum, rd));
    const uint4 c = philox4x32_10(make_uint4(0u, (RNG_ACCEPT << 16) | i, static_cast<uint32_t>(b), stp), k0, k1);
    const float u = bits_to_u01(c.x);
    if (__fmul_rn(u, q) <= p) continue;
    j = i - 1;
    break;
  }
  for (int i = 0; i < j; ++i) out[i] = xb[i];
  s.jmode[2 * b] = j;
  s.jmode[2 * b + 1] = (j < k) ? MODE_RESIDUAL : MODE_BONUS;
}

// Replacement token (residual race, with the log-form race as its fallback) or bonus token.
template <typename T>
__global__ void __launch_bounds__(kThreads) resample_kernel(const T* target, const T* draft, const float* temp, int B,
                                                            int k, int V, Seed seed_arg, const int* step_ptr,
                                                            unsigned step, const unsigned long long* rowkey,
                                                            const unsigned long long* rowsum, int* tokens, int* n,
                                                            AcceptScratch s, int span) {
  pdl_trigger();
  pdl_wait();
  __shared__ unsigned long long red[32];
  __shared__ bool last;
  const int b = blockIdx.x;
  const int mode = s.jmode[2 * b + 1];
  if (mode != MODE_RESIDUAL && mode != MODE_BONUS) return;
  const int j = s.jmode[2 * b];
  const float invT = inv_temp(temp[b]);
  const unsigned stp = step_value(step_ptr, step);
  const unsigned long long seed = seed_value(seed_arg);
  const uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
  const int nt = B * (k + 1);
  const int rt = b * (k + 1) + j;
  const T* trow = target + static_cast<size_t>(rt) * V;
  const bool resid = (mode == MODE_RESIDUAL);
  RowDist dp, dq;
  const T* drow = nullptr;
  if (resid) {
    const int rd = nt + b * k + j;
    dp = row_dist(rowkey, rowsum, rt);
    dq = row_dist(rowkey, rowsum, rd);
    drow = draft + static_cast<size_t>(rd - nt) * V;
  }
  const int lo = blockIdx.y * span, hi = min(V, lo + span);
  unsigned long long best_r = 0, best_l = 0;
  for (int v = lo + threadIdx.x * 4; v < hi; v += kThreads * 4) {
    const uint4 c = philox4x32_10(make_uint4(static_cast<uint32_t>(v >> 2), (RNG_RESAMPLE << 16) | j,
                                             static_cast<uint32_t>(b), stp), k0, k1);
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    float zt[4], zd[4];
    load4<T>(trow, v, zt);
    if (resid) load4<T>(drow, v, zd);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float E = -log_at(bits_to_u01(w[e]));
      const float st = __fmul_rn(zt[e], invT);
      const unsigned long long kl = pack_key(__fsub_rn(st, log_at(E)), v + e);
      best_l = kl > best_l ? kl : best_l;
      if (resid) {
        const float p = __fdiv_rn(exp_cw(__fsub_rn(st, dp.m)), dp.S);
        const float q = __fdiv_rn(exp_cw(__fsub_rn(__fmul_rn(zd[e], invT), dq.m)), dq.S);
        const float r = fmaxf(__fsub_rn(p, q), 0.0f);
        const unsigned long long kr = pack_key(__fdiv_rn(r, E), v + e);
        best_r = kr > best_r ? kr : best_r;
      }
    }
  }
  best_l = block_max_u64(best_l, red);
  best_r = block_max_u64(best_r, red);
  if (threadIdx.x == 0) {
    if (resid) atomicMax(&s.slot[2 * b], best_r);
    atomicMax(&s.slot[2 * b + 1], best_l);
    __threadfence();
    last = (atomicAdd(&s.counter[b], 1) == static_cast<int>(gridDim.y) - 1);
  }
  __syncthreads();
  if (last && threadIdx.x == 0) {
    const unsigned long long r = atomicMax(&s.slot[2 * b], 0ull);
    const unsigned long long l = atomicMax(&s.slot[2 * b + 1], 0ull);
    const bool has_resid = resid && (static_cast<uint32_t>(r >> 32) > 0x80000000u);  // a key > +0
    tokens[static_cast<size_t>(b) * (k + 1) + j] = static_cast<int>(packed_index(has_resid ? r : l));
    n[b] = j + 1;
    s.counter[b] = 0;
  }
}

// One token per row: argmax (T = 0) or the log-form exponential race.
__global__ void __launch_bounds__(kThreads) sample_kernel(const float* logits, long long ld, int V, const float* temp,
                                                          Seed seed_arg, int purpose, int i,
                                                          const int* step_ptr, unsigned step, int* out, int ld_out,
                                                          int* out2, int ld_out2, unsigned long long* slot,
                                                          int* counter, unsigned* err, int span) {
  pdl_trigger();
  pdl_wait();
  __shared__ unsigned long long red[32];
  __shared__ bool last;
  const int b = blockIdx.x;
  const float* row = logits + static_cast<size_t>(b) * ld;
  const float t = temp[b];
  const bool greedy = !(t > 0.f);
  const float invT = greedy ? 1.f : inv_temp(t);
  const unsigned stp = step_value(step_ptr, step);
  const unsigned long long seed = seed_value(seed_arg);
  const uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
  const int lo = blockIdx.y * span, hi = min(V, lo + span);
  unsigned long long best = 0;
  bool bad = false;
  for (int v = lo + threadIdx.x * 4; v < hi; v += kThreads * 4) {
    float z[4];
    load4<float>(row, v, z);
    uint32_t w[4] = {0, 0, 0, 0};
    if (!greedy) {
      const uint4 c = philox4x32_10(make_uint4(static_cast<uint32_t>(v >> 2), (static_cast<uint32_t>(purpose) << 16) | i,
                                               static_cast<uint32_t>(b), stp), k0, k1);
      w[0] = c.x; w[1] = c.y; w[2] = c.z; w[3] = c.w;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      bad |= !isfinite(z[e]);
      float key = z[e];
      if (!greedy) {
        const float E = -log_at(bits_to_u01(w[e]));
        key = __fsub_rn(__fmul_rn(z[e], invT), log_at(E));
      }
      const unsigned long long pk = pack_key(key, v + e);
      best = pk > best ? pk : best;
    }
  }
  best = block_max_u64(best, red);
  if (threadIdx.x == 0) {
    atomicMax(&slot[b], best);
    if (bad) atomicOr(err, static_cast<unsigned>(ERR_NONFINITE));
    __threadfence();
    last = (atomicAdd(&counter[b], 1) == static_cast<int>(gridDim.y) - 1);
  }
  __syncthreads();
  if (last && threadIdx.x == 0) {
    const unsigned long long r = atomicExch(&slot[b], 0ull);
    const int tok = static_cast<int>(packed_index(r));
    out[static_cast<size_t>(b) * ld_out] = tok;
    if (out2) out2[static_cast<size_t>(b) * ld_out2] = tok;
    counter[b] = 0;
  }
}

template <typename T>
cudaError_t accept_typed(const T* target, const T* draft, const int* xhat, const float* temp, int B, int k, int V,
                         Seed seed, unsigned step, const int* step_ptr, const int* stopped, int* tokens,
                         int* n, const AcceptScratch& s, unsigned* err, cudaStream_t st) {
  const int R = B * (2 * k + 1);
  const int span = vocab_span(V, B, 4, kPerCta), S = (V + span - 1) / span;
  const int sspan = vocab_span(V, R, 8, kStatsPerCta), SS = (V + sspan - 1) / sspan;
  // rowkey takes atomic maxima from every CTA of its row, so it is cleared before the first pass;
  // rowsum (placed after the rowkey of the scratch's own batch size, which may exceed B) is cleared
  // by the first pass itself
  cudaError_t e = cudaMemsetAsync(s.rowkey, 0, sizeof(unsigned long long) * R, st);
  if (e != cudaSuccess) return e;
  { const cudaError_t e_ = launch_pdl(rowmax_kernel<T>, dim3(dim3(R, SS)), dim3(kThreads), 0, st, target, draft, B, k, V, temp, stopped, s.rowkey, s.rowsum, err, sspan); if (e_ != cudaSuccess) return e_; }
  { const cudaError_t e_ = launch_pdl(rowsum_kernel<T>, dim3(dim3(R, SS)), dim3(kThreads), 0, st, target, draft, B, k, V, temp, stopped, s.rowkey, s.rowsum, sspan); if (e_ != cudaSuccess) return e_; }
  { const cudaError_t e_ = launch_pdl(decide_kernel<T>, dim3((B + 127) / 128), dim3(128), 0, st, target, draft, xhat, temp, B, k, V, seed, step_ptr, step, stopped,
                                                    s.rowkey, s.rowsum, tokens, n, s); if (e_ != cudaSuccess) return e_; }
  { const cudaError_t e_ = launch_pdl(resample_kernel<T>, dim3(dim3(B, S)), dim3(kThreads), 0, st, target, draft, temp, B, k, V, seed, step_ptr, step, s.rowkey,
                                                      s.rowsum, tokens, n, s, span); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

}  // namespace

size_t accept_scratch_bytes(int B, int k) {
  const size_t R = static_cast<size_t>(B) * (2 * k + 1);
  return 8 * (2 * R) + 8 * (2 * static_cast<size_t>(B)) + 4 * static_cast<size_t>(B) + 4 * 2 * static_cast<size_t>(B) + 64;
}

AcceptScratch accept_scratch_carve(void* base, int B, int k) {
  const size_t R = static_cast<size_t>(B) * (2 * k + 1);
  AcceptScratch s;
  unsigned long long* p = static_cast<unsigned long long*>(base);
  s.rowkey = p;
  s.rowsum = p + R;
  s.slot = p + 2 * R;
  s.counter = reinterpret_cast<int*>(p + 2 * R + 2 * B);
  s.jmode = s.counter + B;
  return s;
}

cudaError_t accept_blocks(const void* target, const void* draft, int dtype, const int* xhat, const float* temp, int B,
                          int k, int V, Seed seed, unsigned step, const int* step_ptr, const int* stopped,
                          int* tokens, int* n, const AcceptScratch& s, unsigned* err, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  if (dtype == 1)
    return accept_typed<bf16>(static_cast<const bf16*>(target), static_cast<const bf16*>(draft), xhat, temp, B, k, V,
                              seed, step, step_ptr, stopped, tokens, n, s, err, st);
  return accept_typed<float>(static_cast<const float*>(target), static_cast<const float*>(draft), xhat, temp, B, k, V,
                             seed, step, step_ptr, stopped, tokens, n, s, err, st);
}

cudaError_t sample_rows(const float* logits, long long ld, int B, int V, const float* temp, Seed seed,
                        int purpose, int i, const int* step_ptr, unsigned step, int* out, int ld_out, int* out2,
                        int ld_out2, unsigned long long* slot, int* counter, unsigned* err, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  const int span = vocab_span(V, B, 4, kPerCta), S = (V + span - 1) / span;
  { const cudaError_t e_ = launch_pdl(sample_kernel, dim3(dim3(B, S)), dim3(kThreads), 0, st, logits, ld, V, temp, seed, purpose, i, step_ptr, step, out, ld_out,
                                                 out2, ld_out2, slot, counter, err, span); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

}  // namespace sd2
