// Causal attention over the paged KV cache, grouped by sequence (verifier block of k+1 rows,
// drafter rows, or prompt rows) and by KV head (grouped-query attention).
//
// One CTA = (row group of one sequence, KV head, split of the context). It stages the split's
// K and V in 64-position tiles in shared memory (rows padded by 16 bytes so that the per-lane
// 16-byte reads of eight lanes hit distinct banks), and each warp runs an online softmax for up
// to 8 query vectors (query rows x the heads sharing the KV head). Every K/V byte of the split
// is read from HBM once per CTA, whatever the number of rows in the group. With several splits
// each CTA stores its partial (max, sum, accumulator) triples, and the last CTA of the
// (group, KV head) to arrive merges them in split order.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace sd2 {
namespace {

constexpr int kTile = 64;
constexpr int kWarps = 8;
constexpr int kQPW = 8;               // query vectors per warp
constexpr int kMaxQV = kWarps * kQPW;  // per CTA
constexpr int kMaxMergeSplits = 64;     // context splits one merge handles (weights in smem)

template <int HD>
constexpr int smem_bytes() {
  return (2 * kTile * (HD + 8) * 2 + kMaxQV * HD * 4) > (2 * kMaxQV * kMaxMergeSplits * 4)
             ? (2 * kTile * (HD + 8) * 2 + kMaxQV * HD * 4)
             : (2 * kMaxQV * kMaxMergeSplits * 4);
}

template <int HD>
__global__ void __launch_bounds__(kWarps * 32) attn_kernel(const AttnArgs a) {
  pdl_trigger();
  pdl_wait();
  constexpr int DPL = HD / 32;        // output dims per lane
  constexpr int KS = HD + 8;          // padded smem row (bf16 elements)
  extern __shared__ __align__(16) unsigned char smem[];
  bf16* sK = reinterpret_cast<bf16*>(smem);
  bf16* sV = sK + kTile * KS;
  float* sQ = reinterpret_cast<float*>(sV + kTile * KS);

  const int g = blockIdx.x, kvh = blockIdx.y, split = blockIdx.z;
  const int r0 = a.grp_row0[g], nr = a.grp_nrows[g], seq = a.grp_seq[g];
  const int Hkv = a.kv.Hkv, G = a.H / Hkv;
  const int nqv = nr * G;
  int pmax = 0;
  for (int i = 0; i < nr; ++i) pmax = max(pmax, a.row_pos[r0 + i]);
  const int lo = split * a.chunk;
  if (lo > pmax) return;
  const int hi = min(lo + a.chunk, pmax + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // queries of the group -> shared memory
  for (int idx = threadIdx.x; idx < nqv * (HD / 4); idx += blockDim.x) {
    const int qv = idx / (HD / 4), c = idx % (HD / 4);
    const int row = r0 + qv / G, h = kvh * G + qv % G;
    reinterpret_cast<float4*>(sQ)[qv * (HD / 4) + c] =
        reinterpret_cast<const float4*>(a.q + (static_cast<size_t>(row) * a.H + h) * HD)[c];
  }

  float m_run[kQPW], l_run[kQPW], acc[kQPW][DPL];
  int pos_r[kQPW];
#pragma unroll
  for (int j = 0; j < kQPW; ++j) {
    m_run[j] = -INFINITY;
    l_run[j] = 0.f;
#pragma unroll
    for (int d = 0; d < DPL; ++d) acc[j][d] = 0.f;
    const int qv = warp + kWarps * j;
    pos_r[j] = qv < nqv ? a.row_pos[r0 + qv / G] : -1;
  }
  const float scale = rsqrtf(static_cast<float>(HD));
  const bf16* pool = static_cast<const bf16*>(a.kv.pool);
  const size_t head_stride = static_cast<size_t>(16) * HD;
  const size_t blk_stride = static_cast<size_t>(2) * Hkv * head_stride;
  const int* table = a.kv.table + static_cast<size_t>(seq) * a.kv.bt_stride;

  for (int t0 = lo; t0 < hi; t0 += kTile) {
    __syncthreads();
    // stage K and V rows t0 .. t0+63 (zeros beyond hi)
    constexpr int CPR = HD / 8;  // 16-byte chunks per row
    for (int idx = threadIdx.x; idx < kTile * CPR; idx += blockDim.x) {
      const int t = idx / CPR, c = idx % CPR;
      const int p = t0 + t;
      uint4 kvk = make_uint4(0, 0, 0, 0), kvv = make_uint4(0, 0, 0, 0);
      if (p < hi) {
        const int blk = table[p >> 4];
        const bf16* base = pool + (static_cast<size_t>(a.layer) * a.kv.n_blocks + blk) * blk_stride +
                           kvh * head_stride + (p & 15) * HD;
        kvk = __ldg(reinterpret_cast<const uint4*>(base) + c);
        kvv = __ldg(reinterpret_cast<const uint4*>(base + Hkv * head_stride) + c);
      }
      *reinterpret_cast<uint4*>(sK + t * KS + c * 8) = kvk;
      *reinterpret_cast<uint4*>(sV + t * KS + c * 8) = kvv;
    }
    __syncthreads();

#pragma unroll
    for (int j = 0; j < kQPW; ++j) {
      const int qv = warp + kWarps * j;
      if (qv >= nqv) break;
      if (pos_r[j] < t0) continue;  // whole tile after this row's position
      const float* q = sQ + qv * HD;
      float s0 = 0.f, s1 = 0.f;
#pragma unroll 4
      for (int c = 0; c < HD / 8; ++c) {
        const float4 qa = reinterpret_cast<const float4*>(q)[2 * c];
        const float4 qb = reinterpret_cast<const float4*>(q)[2 * c + 1];
        const uint4 k0 = *reinterpret_cast<const uint4*>(sK + lane * KS + c * 8);
        const uint4 k1 = *reinterpret_cast<const uint4*>(sK + (lane + 32) * KS + c * 8);
        s0 = fmaf(qa.x, bf_lo(k0.x), s0); s0 = fmaf(qa.y, bf_hi(k0.x), s0);
        s0 = fmaf(qa.z, bf_lo(k0.y), s0); s0 = fmaf(qa.w, bf_hi(k0.y), s0);
        s0 = fmaf(qb.x, bf_lo(k0.z), s0); s0 = fmaf(qb.y, bf_hi(k0.z), s0);
        s0 = fmaf(qb.z, bf_lo(k0.w), s0); s0 = fmaf(qb.w, bf_hi(k0.w), s0);
        s1 = fmaf(qa.x, bf_lo(k1.x), s1); s1 = fmaf(qa.y, bf_hi(k1.x), s1);
        s1 = fmaf(qa.z, bf_lo(k1.y), s1); s1 = fmaf(qa.w, bf_hi(k1.y), s1);
        s1 = fmaf(qb.x, bf_lo(k1.z), s1); s1 = fmaf(qb.y, bf_hi(k1.z), s1);
        s1 = fmaf(qb.z, bf_lo(k1.w), s1); s1 = fmaf(qb.w, bf_hi(k1.w), s1);
      }
      const int p0 = t0 + lane, p1 = t0 + lane + 32;
      s0 = (p0 < hi && p0 <= pos_r[j]) ? s0 * scale : -INFINITY;
      s1 = (p1 < hi && p1 <= pos_r[j]) ? s1 * scale : -INFINITY;
      const float mt = warp_max(fmaxf(s0, s1));
      const float m_new = fmaxf(m_run[j], mt);
      const float corr = __expf(m_run[j] - m_new);
      const float e0 = __expf(s0 - m_new), e1 = __expf(s1 - m_new);
      l_run[j] = l_run[j] * corr + warp_sum(e0 + e1);
      m_run[j] = m_new;
#pragma unroll
      for (int d = 0; d < DPL; ++d) acc[j][d] *= corr;
      const int tmax = min(32, hi - t0);
      for (int t = 0; t < tmax; ++t) {
        const float w0 = __shfl_sync(0xffffffffu, e0, t);
        const float w1 = __shfl_sync(0xffffffffu, e1, t);
        const bf16* v0 = sV + t * KS + lane * DPL;
        const bf16* v1 = sV + (t + 32) * KS + lane * DPL;
#pragma unroll
        for (int d = 0; d < DPL; ++d)
          acc[j][d] = fmaf(w0, bf2f(v0[d]), fmaf(w1, bf2f(v1[d]), acc[j][d]));
      }
    }
  }

#pragma unroll
  for (int j = 0; j < kQPW; ++j) {
    const int qv = warp + kWarps * j;
    if (qv >= nqv) break;
    const int row = r0 + qv / G, h = kvh * G + qv % G;
    if (a.n_splits == 1) {
      const float inv = 1.f / l_run[j];
      bf16* o = static_cast<bf16*>(a.out) + static_cast<size_t>(row) * a.H * HD + h * HD + lane * DPL;
#pragma unroll
      for (int d = 0; d < DPL; ++d) o[d] = __float2bfloat16_rn(acc[j][d] * inv);
    } else {
      float* p = a.part + ((static_cast<size_t>(row) * a.H + h) * a.n_splits + split) * (HD + 2);
      if (lane == 0) { p[0] = m_run[j]; p[1] = l_run[j]; }
#pragma unroll
      for (int d = 0; d < DPL; ++d) p[2 + lane * DPL + d] = acc[j][d];
    }
  }
  if (a.n_splits == 1) return;

  // The splits that run for this group are those starting at or before its last position.
  __shared__ int last_flag;
  __syncthreads();
  if (threadIdx.x == 0) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;"
                 : "=r"(old)
                 : "l"(a.counters + static_cast<size_t>(g) * Hkv + kvh)
                 : "memory");
    const int n_used = pmax / a.chunk + 1;
    last_flag = (old == n_used - 1) ? 1 : 0;
    if (last_flag) a.counters[static_cast<size_t>(g) * Hkv + kvh] = 0;
  }
  __syncthreads();
  if (!last_flag) return;
  // merge: out = sum_s acc_s e^{m_s - M} / sum_s l_s e^{m_s - M} for every (row, head) here.
  // (1) every thread gathers (m_s, l_s) pairs into shared memory, (2) one thread per query
  // vector turns them into split weights, (3) all threads form the weighted sums over hd with
  // coalesced loads. At most kMaxMergeSplits splits, so the weights fit in shared memory.
  float* sW = reinterpret_cast<float*>(smem);               // [kMaxQV][n_splits] weights
  float* sL = sW + kMaxQV * kMaxMergeSplits;                 // [kMaxQV][n_splits] sums
  const int NS = a.n_splits;
  for (int idx = threadIdx.x; idx < nqv * NS; idx += blockDim.x) {
    const int qv = idx / NS, s2 = idx % NS;
    const int row = r0 + qv / G, h = kvh * G + qv % G;
    const int ns = min(NS, a.row_pos[row] / a.chunk + 1);
    const float* ps = a.part + ((static_cast<size_t>(row) * a.H + h) * NS + s2) * (HD + 2);
    sW[qv * NS + s2] = s2 < ns ? __ldcg(ps) : -INFINITY;
    sL[qv * NS + s2] = s2 < ns ? __ldcg(ps + 1) : 0.f;
  }
  __syncthreads();
  if (threadIdx.x < nqv) {
    const int qv = threadIdx.x;
    float M = -INFINITY;
    for (int s2 = 0; s2 < NS; ++s2) M = fmaxf(M, sW[qv * NS + s2]);
    float L = 0.f;
    for (int s2 = 0; s2 < NS; ++s2) {
      const float w = __expf(sW[qv * NS + s2] - M);          // exp(-inf) = 0 for absent splits
      sW[qv * NS + s2] = w;
      L += sL[qv * NS + s2] * w;
    }
    const float inv = 1.f / L;
    for (int s2 = 0; s2 < NS; ++s2) sW[qv * NS + s2] *= inv;
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < nqv * HD; idx += blockDim.x) {
    const int qv = idx / HD, d = idx % HD;
    const int row = r0 + qv / G, h = kvh * G + qv % G;
    const int ns = min(NS, a.row_pos[row] / a.chunk + 1);
    const float* p = a.part + (static_cast<size_t>(row) * a.H + h) * NS * (HD + 2) + 2 + d;
    float o = 0.f;
#pragma unroll 4
    for (int s2 = 0; s2 < ns; ++s2) o += sW[qv * NS + s2] * __ldcg(p + static_cast<size_t>(s2) * (HD + 2));
    static_cast<bf16*>(a.out)[static_cast<size_t>(row) * a.H * HD + h * HD + d] = __float2bfloat16_rn(o);
  }
}


template <int HD>
cudaError_t launch(const AttnArgs& a, cudaStream_t st) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<HD>());
    if (e != cudaSuccess) return e;
    configured = true;
  }
  dim3 grid(a.n_groups, a.kv.Hkv, a.n_splits);
  { const cudaError_t e_ = launch_pdl(attn_kernel<HD>, dim3(grid), dim3(kWarps * 32), smem_bytes<HD>(), st, a); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

}  // namespace

cudaError_t attention(const AttnArgs& a, cudaStream_t st) {
  if (a.n_groups <= 0) return cudaSuccess;
  if (a.n_splits > kMaxMergeSplits || a.chunk % kTile != 0) return cudaErrorInvalidValue;
  if (a.hd == 128) return launch<128>(a, st);
  if (a.hd == 64) return launch<64>(a, st);
  return cudaErrorInvalidValue;
}

}  // namespace sd2
