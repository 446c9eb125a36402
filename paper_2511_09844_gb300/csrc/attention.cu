// Causal attention over the paged KV cache, grouped by sequence (verifier block of k+1 rows,
// drafter rows, or prompt rows) and by KV head (grouped-query attention).
//
// One CTA = (split of the context, row group of one sequence, KV head). Its query vectors (query
// rows x the heads sharing the KV head, at most 64) are the M side of two small contractions per
// 64-position tile, both on the tensor cores with mma.sync m16n8k16 (bf16 in, f32 accumulate):
//   scores S = Q K^T      warp w owns positions 8w .. 8w+7 of the tile, every query tile
//   online softmax        4 threads per query row: running max/sum, P = e^{S - m} in bf16
//   O = O * corr + P V    warp w owns 8 (hd 64) or 16 (hd 128) output dimensions
// The contractions are tiny (M <= 64); the kernel is bound by the latency of its loads, so they
// are ordered by when their data is final. The block ids of the split are read before the
// programmatic wait (they are fixed before the step starts). In a decode step the cache positions
// below the sequence's pre-step length were also written before the step: their K/V rows are
// requested before the wait, and the few rows the step itself may have written are requested
// right after it, together with the queries and row positions. K/V tiles are staged with
// cp.async (zero-filled where no row exists) through a ring of 2 to 4 tiles (the launcher takes
// the deepest ring that keeps the grid resident); every K/V byte of the split is read from HBM
// once per CTA.
//
// The splits of one (row group, KV head) form a thread-block cluster. Split merge: the (query
// vector, 4 dimensions) elements of the group are shared out over the splits; every split pushes
// its running max and sum of each query vector to every split, and each accumulator pair to the
// split owning its element, with asynchronous stores that complete on the owner's receive
// mbarrier. The owner waits only for its own share, merges it and writes the output; no partial
// goes through global memory and no cluster barrier is held while the partials travel. Where
// two CTAs per SM fit only that way, the receive buffers lie over the K/V ring: each split then
// arrives on the cluster barrier after its last tile, so no partial lands in a ring still read.
// Long contexts add clusters along the context whose owners meet through global partials; decode
// steps over many ragged sequences run in flat mode (one-CTA clusters shared out by length on the
// device, global partials, the last split of a sequence merging).
#include <limits.h>
#include <math.h>

#include <array>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace sd2 {
namespace {

constexpr int kTile = 64;               // positions per K/V tile
constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kMaxQV = 64;              // query vectors per CTA
constexpr int kMaxSplits = 16;          // context splits = CTAs of one cluster (16: non-portable size)
constexpr int kMaxSmem = 200 * 1024;   // dynamic shared memory opt-in (static arrays come on top)
constexpr int kMaxBuf = 4;             // K/V tiles of the ring
constexpr int kFlatMaxSplits = 32;     // slots one row group takes in flat mode
// Resident CTAs per SM the register budget allows: hd = 64 fits 64 registers a thread, so four
// CTAs; hd = 128 keeps two.
template <int HD>
constexpr int kCtasPerSm = HD == 64 ? 4 : 2;

template <int HD>
struct AttnCfg {
  static constexpr int KS = HD + 8;                     // Q/K/V row stride, bf16 (conflict-free fragments)
  static constexpr int SS = kTile + 8;                  // score row stride, f32
  static constexpr int PS = kTile + 8;                  // probability row stride, bf16
  static constexpr int ROW_BYTES = 4 * kMaxQV * 4;      // per query vector: position, correction, max, sum
  static constexpr int KV_TILE = 2 * kTile * KS * 2;    // K and V of one tile
  __host__ __device__ static int qrows(int max_rows, int G) {
    const int r = ((max_rows * G + 15) / 16) * 16;
    return r < kMaxQV ? r : kMaxQV;
  }
  // layout: row data, Q, S, P, a ring of nb K/V tiles, the split's block ids; split merge (ns > 1):
  // receive barrier, every split's (max, sum) per query vector [ns][qr] and every split's
  // accumulators of this rank's share of elements [ns][share] (float4 each), after the block ids
  // or, with `ring`, over the K/V ring
  __host__ __device__ static size_t q_off() { return ROW_BYTES; }
  __host__ __device__ static size_t s_off(int qr) { return q_off() + static_cast<size_t>(qr) * KS * 2; }
  __host__ __device__ static size_t p_off(int qr) { return s_off(qr) + static_cast<size_t>(qr) * SS * 4; }
  __host__ __device__ static size_t kv_off(int qr) { return p_off(qr) + static_cast<size_t>(qr) * PS * 2; }
  __host__ __device__ static size_t blk_off(int qr, int nb) { return kv_off(qr) + static_cast<size_t>(nb) * KV_TILE; }
  __host__ __device__ static int share(int qr, int ns) { return (qr * (HD / 4) + ns - 1) / ns; }
  __host__ __device__ static size_t rcv_off(int qr, int chunk, int nb) {
    return blk_off(qr, nb) + ((static_cast<size_t>(chunk / 16) * 4 + 15) & ~static_cast<size_t>(15));
  }
  __host__ __device__ static size_t ml_off(int qr, int chunk, int nb, int ring) {
    return ring ? kv_off(qr) : rcv_off(qr, chunk, nb) + 16;
  }
  __host__ __device__ static size_t acc_off(int qr, int chunk, int nb, int ring, int ns) {
    return ml_off(qr, chunk, nb, ring) + static_cast<size_t>(ns) * qr * 8;
  }
  static size_t merge_bytes(int qr, int ns) {
    return static_cast<size_t>(ns) * qr * 8 + static_cast<size_t>(ns) * share(qr, ns) * 16;
  }
  static size_t bytes(int qr, int chunk, int ns, int nb, int ring) {
    if (ns == 1) return rcv_off(qr, chunk, nb);
    return ring ? rcv_off(qr, chunk, nb) + 16 : acc_off(qr, chunk, nb, 0, ns) + static_cast<size_t>(ns) * share(qr, ns) * 16;
  }
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint32_t pack_bf2(float x, float y) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }
// wait until at most n (0..3) of this thread's most recent cp.async groups are pending
__device__ __forceinline__ void cp_async_wait_n(int n) {
  if (n <= 0) cp_async_wait<0>();
  else if (n == 1) cp_async_wait<1>();
  else if (n == 2) cp_async_wait<2>();
  else cp_async_wait<3>();
}
// two fp32 stored asynchronously to `raddr` (shared::cluster, 8-byte aligned), completing 8 bytes
// of a transaction on the mbarrier at `rbar` (shared::cluster, same CTA)
__device__ __forceinline__ void st_async_v2(uint32_t raddr, uint32_t rbar, float x, float y) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(raddr),
               "f"(x), "f"(y), "r"(rbar)
               : "memory");
}

// D(16x8, f32) += A(16x16, bf16, row-major) * B(16x8, bf16, column-major)
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
__device__ __forceinline__ void ldsm_x2_t(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(addr)
               : "memory");
}

// Context clusters (R > 1): the cluster's owner of an element share writes its unnormalised partial
// (sum over its splits of e^{m_s - M_r} acc_s, with M_r and L_r = sum e^{m_s - M_r} l_s) to global
// scratch, then counts itself in with a self-resetting atomicInc; the last of the R owners of the
// share combines the R partials (max, weights e^{M_r - M}, normaliser, in cluster order) and writes
// the output. No CTA waits for another.
template <int HD>
__device__ void ctx_cluster_merge(const AttnArgs& a, const float2* rML, const float4* rAcc, int QR, int share,
                                  int e_lo, int e_hi, int g, int kvh, int rank, int cr, int R, int r0, int G,
                                  int* sLast) {
  const int NS = a.n_splits, Hkv = a.kv.Hkv, tid = threadIdx.x;
  constexpr int E4MAX = kMaxQV * (HD / 4);                          // partial slots per (group, KV head, cluster)
  float4* pacc = static_cast<float4*>(a.part_acc);
  float2* pml = static_cast<float2*>(a.part_ml);
  const size_t base = (static_cast<size_t>(g) * Hkv + kvh) * R * E4MAX;
  for (int e = e_lo + tid; e < e_hi; e += kThreads) {
    const int qv = e / (HD / 4);
    float M = -INFINITY;
    for (int s2 = 0; s2 < NS; ++s2) M = fmaxf(M, rML[s2 * QR + qv].x);
    const float Mu = M == -INFINITY ? 0.f : M;                      // a cluster no row can see
    float L = 0.f;
    float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s2 = 0; s2 < NS; ++s2) {                               // in split order
      const float2 ml = rML[s2 * QR + qv];
      const float w = __expf(ml.x - Mu);
      const float4 v = rAcc[s2 * share + (e - e_lo)];
      L = fmaf(ml.y, w, L);
      o.x = fmaf(w, v.x, o.x); o.y = fmaf(w, v.y, o.y);
      o.z = fmaf(w, v.z, o.z); o.w = fmaf(w, v.w, o.w);
    }
    pacc[base + static_cast<size_t>(cr) * E4MAX + e] = o;
    pml[base + static_cast<size_t>(cr) * E4MAX + e] = make_float2(M, L);
  }
  __threadfence();                                                  // the partials before the count
  __syncthreads();
  if (tid == 0) {
    unsigned* cnt = static_cast<unsigned*>(a.part_cnt) + (static_cast<size_t>(g) * Hkv + kvh) * NS + rank;
    *sLast = atomicInc(cnt, static_cast<unsigned>(R - 1)) == static_cast<unsigned>(R - 1) ? 1 : 0;
  }
  __syncthreads();
  if (!*sLast) return;
  __threadfence();                                                  // every cluster's partials are visible
  for (int e = e_lo + tid; e < e_hi; e += kThreads) {
    const int qv = e / (HD / 4), d4 = e % (HD / 4);
    float M = -INFINITY;
    for (int q = 0; q < R; ++q) M = fmaxf(M, __ldcg(&pml[base + static_cast<size_t>(q) * E4MAX + e]).x);
    float L = 0.f;
    float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int q = 0; q < R; ++q) {
      const float2 ml = __ldcg(&pml[base + static_cast<size_t>(q) * E4MAX + e]);
      const float4 v = __ldcg(&pacc[base + static_cast<size_t>(q) * E4MAX + e]);
      const float w = ml.x == -INFINITY ? 0.f : __expf(ml.x - M);
      L = fmaf(ml.y, w, L);
      o.x = fmaf(w, v.x, o.x); o.y = fmaf(w, v.y, o.y);
      o.z = fmaf(w, v.z, o.z); o.w = fmaf(w, v.w, o.w);
    }
    const float inv = 1.f / L;
    const size_t rh = static_cast<size_t>(r0 + qv / G) * a.H + kvh * G + qv % G;
    *reinterpret_cast<uint2*>(static_cast<bf16*>(a.out) + rh * HD + d4 * 4) =
        make_uint2(pack_bf2(o.x * inv, o.y * inv), pack_bf2(o.z * inv, o.w * inv));
  }
}

// NB: K/V tiles of the shared-memory layout (>= 2 when a.chunk > 64); ring: the split-merge
// receive buffers lie over the K/V ring (n_splits > 1). DEC: 1 for a decode step with one
// context cluster per (group, KV head) and separate merge buffers (the batch-1 steps), whose
// instantiation then carries none of the other paths' code; 0 decides everything at run time.
template <int HD, int DEC>
__global__ void __launch_bounds__(kThreads, kCtasPerSm<HD>) attn_kernel(const AttnArgs a, int NB, int ring_arg) {
  using C = AttnCfg<HD>;
  constexpr int KS = C::KS, SS = C::SS, PS = C::PS;
  constexpr int NT = HD / 64;  // n8 tiles of output dimensions per warp
  pdl_trigger();
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int sPmax[2];
  __shared__ int sRecv;

  // x = context cluster r (of R) x rank in the cluster: split = blockIdx.x orders the context
  // ranges, rank = the CTA's place in its cluster (its merge share)
  int split = blockIdx.x, g = blockIdx.y;
  const int kvh = blockIdx.z;
  const int NS = a.n_splits, R = DEC ? 1 : (a.n_ctx_clusters > 1 ? a.n_ctx_clusters : 1);
  const int ring = DEC ? 0 : ring_arg;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // Flat mode: slot blockIdx.x of this KV head -> (group g, split of Rf). Group j takes
  // ceil(tiles_j / t) slots, tiles_j its visible length in 64-position tiles and t the smallest
  // count for which all groups fit the slots, so no slot holds more than t tiles; slots past the
  // last group have nothing to do. Every CTA derives the same map from the pre-step lengths.
  int Rf = 1, slot0 = 0;
  if (!DEC && a.flat > 0) {
    __shared__ int sMap[3];
    if (warp == 0) {
      const int ng = a.n_groups, W = a.flat;
      auto tiles_of = [&](int j) {
        const int L = a.pre_len[a.grp_seq[j]] + a.pre_stable + a.pre_fresh;
        return max(1, (L + kTile - 1) / kTile);
      };
      const int t0 = lane < ng ? tiles_of(lane) : 0, t1 = lane + 32 < ng ? tiles_of(lane + 32) : 0;
      const int T = __reduce_add_sync(0xffffffffu, t0 + t1);
      const int tmax = __reduce_max_sync(0xffffffffu, max(t0, t1));
      // at most kFlatMaxSplits slots a group (the merge stages their weights in shared memory)
      int t_lo = max(max(1, (T + W - 1) / W), (tmax + kFlatMaxSplits - 1) / kFlatMaxSplits), t_hi = max(t_lo, tmax);
      while (t_lo < t_hi) {                          // warp-uniform bisection
        const int t = (t_lo + t_hi) >> 1;
        const int need = __reduce_add_sync(0xffffffffu, (t0 + t - 1) / t + (t1 + t - 1) / t);
        if (need <= W) t_hi = t; else t_lo = t + 1;
      }
      const int n0 = (t0 + t_lo - 1) / t_lo, n1 = (t1 + t_lo - 1) / t_lo;
      int p0 = n0, p1 = n1;                          // inclusive prefix sums over groups 0..31, 32..63
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int v0 = __shfl_up_sync(0xffffffffu, p0, off), v1 = __shfl_up_sync(0xffffffffu, p1, off);
        if (lane >= off) { p0 += v0; p1 += v1; }
      }
      p1 += __shfl_sync(0xffffffffu, p0, 31);
      const int sl = blockIdx.x;
      const bool in0 = lane < ng && sl >= p0 - n0 && sl < p0;
      const bool in1 = lane + 32 < ng && sl >= p1 - n1 && sl < p1;
      if (lane == 0) sMap[0] = -1;
      __syncwarp();
      if (in0) { sMap[0] = lane; sMap[1] = p0 - n0; sMap[2] = n0; }
      if (in1) { sMap[0] = lane + 32; sMap[1] = p1 - n1; sMap[2] = n1; }
    }
    __syncthreads();
    g = sMap[0];
    if (g < 0) return;                               // a slot past the last group
    slot0 = sMap[1];
    Rf = sMap[2];
    split = blockIdx.x - slot0;
  }
  const int rank = split % NS, cr = split / NS;
  const int g8 = lane >> 2, t4 = lane & 3;
  const int Hkv = a.kv.Hkv, G = a.H / Hkv;
  const int QR = C::qrows(a.max_rows, G);
  int* sPos = reinterpret_cast<int*>(smem);
  float* sCorr = reinterpret_cast<float*>(smem) + kMaxQV;
  float* sL = sCorr + 2 * kMaxQV;
  bf16* sQ = reinterpret_cast<bf16*>(smem + C::q_off());
  float* sS = reinterpret_cast<float*>(smem + C::s_off(QR));
  bf16* sP = reinterpret_cast<bf16*>(smem + C::p_off(QR));
  unsigned char* sKV = smem + C::kv_off(QR);
  int* sBlk = reinterpret_cast<int*>(smem + C::blk_off(QR, NB));
  const uint32_t rbar = smem_u32(smem + C::rcv_off(QR, a.chunk, NB));
  const float2* rML = reinterpret_cast<const float2*>(smem + C::ml_off(QR, a.chunk, NB, ring));
  const float4* rAcc = reinterpret_cast<const float4*>(smem + C::acc_off(QR, a.chunk, NB, ring, NS));
  const int share = C::share(QR, NS);

  // Before the wait: the plan tables and the block table (written before the step's first
  // kernel) and, in a decode step, the sequence's pre-step length.
  const int r0 = a.grp_row0[g], nr = a.grp_nrows[g], seq = a.grp_seq[g];
  const int nqv = nr * G;
  // A decode step knows, before the wait, that its rows lie below len + pre_stable + pre_fresh: the
  // splits share that range (whole tiles, at most a.chunk each) instead of the planned maximum, so
  // no split is empty while another holds several tiles.
  const bool early = DEC ? true : a.pre_len != nullptr;
  const int len = early ? a.pre_len[seq] : 0;
  int chunk = a.chunk;
  if (early) {
    const int per = (len + a.pre_stable + a.pre_fresh + NS * R * Rf - 1) / (NS * R * Rf);
    chunk = min(a.chunk, max(kTile, ((per + kTile - 1) / kTile) * kTile));
  }
  const int lo = split * chunk;
  const int nblk = min(chunk >> 4, a.kv.bt_stride - (lo >> 4));
  const int row_end = lo + nblk * 16;               // positions the split's block ids cover
  {
    const int* table = a.kv.table + static_cast<size_t>(seq) * a.kv.bt_stride + (lo >> 4);
    for (int i = tid; i < nblk; i += kThreads) sBlk[i] = table[i];
  }
  int pre_hi = lo, fresh_hi = lo;                   // rows [lo, pre_hi) early, [pre_hi, fresh_hi) after the wait
  if (early) {
    pre_hi = min(max(lo, len + a.pre_stable), row_end);
    fresh_hi = min(max(pre_hi, len + a.pre_stable + a.pre_fresh), row_end);
  }
  const int E4 = nqv * (HD / 4);                    // merge elements: (query vector, 4 dimensions)
  const int e_lo = rank * E4 / NS, e_hi = (rank + 1) * E4 / NS;
  if (NS > 1 && tid == 0) {
    tc::mbar_init(rbar, 1);
    tc::mbar_expect_tx(rbar, static_cast<uint32_t>(NS * ((e_hi - e_lo) * 16 + nqv * 8)));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();                                  // block ids and the receive barrier
  if (NS > 1 && !ring) cluster_arrive_relaxed();    // waited for before the first push

  const bf16* pool = static_cast<const bf16*>(a.kv.pool);
  const size_t head_stride = static_cast<size_t>(16) * HD;
  const size_t blk_stride = static_cast<size_t>(2) * Hkv * head_stride;
  const bf16* layer_base = pool + static_cast<size_t>(a.layer) * a.kv.n_blocks * blk_stride + kvh * head_stride;
  // ring slots used (the dynamic chunk may hold fewer tiles than the layout)
  const int nb = chunk > kTile ? max(2, min(NB, chunk / kTile)) : 1;
  // rows p in [p_from, p_to) of tile i (positions lo + 64 i ..) -> ring slot i % nb: loaded below
  // `valid_end`, zero-filled from it on
  auto issue_rows = [&](int i, int p_from, int p_to, int valid_end) {
    bf16* dK = reinterpret_cast<bf16*>(sKV + (i % nb) * C::KV_TILE);
    bf16* dV = dK + kTile * KS;
    const int t0 = lo + i * kTile;
#pragma unroll
    for (int u = 0; u < kTile * (HD / 8) / kThreads; ++u) {
      const int idx = tid + u * kThreads, t = idx / (HD / 8), c = idx % (HD / 8);
      const int p = t0 + t;
      if (p < p_from || p >= p_to) continue;
      const bool ok = p < valid_end && p < row_end;   // block ids exist only below row_end
      const bf16* src = layer_base;
      if (ok) src += static_cast<size_t>(sBlk[(p - lo) >> 4]) * blk_stride + static_cast<size_t>(p & 15) * HD + c * 8;
      cp_async16(smem_u32(dK + t * KS + c * 8), src, ok);
      cp_async16(smem_u32(dV + t * KS + c * 8), ok ? src + Hkv * head_stride : layer_base, ok);
    }
  };
  if (early)
    for (int i = 0; i < nb; ++i) issue_rows(i, lo, pre_hi, pre_hi);
  pdl_wait();
  if (early)   // the rows this step may have written, beside the queries
    for (int i = 0; i < nb; ++i) {
      issue_rows(i, pre_hi, INT_MAX, fresh_hi);
      cp_async_commit();
    }
  int pq = -1;
  if (tid < nqv) pq = __ldcg(a.row_pos + r0 + tid / G);
  constexpr int QC = HD / 4;                        // float4 per query vector
  constexpr int QPT = kMaxQV * QC / kThreads;
  float4 qr[QPT];
#pragma unroll
  for (int u = 0; u < QPT; ++u) {
    const int idx = tid + u * kThreads, qv = idx / QC, c = idx % QC;
    qr[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (qv < nqv)
      qr[u] = __ldcg(reinterpret_cast<const float4*>(
                         a.q + (static_cast<size_t>(r0 + qv / G) * a.H + kvh * G + qv % G) * HD) + c);
  }
  if (tid < kMaxQV) sPos[tid] = pq;
#pragma unroll
  for (int u = 0; u < QPT; ++u) {
    const int idx = tid + u * kThreads, qv = idx / QC, c = idx % QC;
    if (qv < QR)
      *reinterpret_cast<uint2*>(sQ + qv * KS + c * 4) =
          make_uint2(pack_bf2(qr[u].x, qr[u].y), pack_bf2(qr[u].z, qr[u].w));
  }
  const int wmax = __reduce_max_sync(0xffffffffu, pq);
  if (warp < 2 && lane == 0) sPmax[warp] = wmax;
  __syncthreads();
  const int pmax = max(sPmax[0], sPmax[1]);
  // A split that starts after every row of the group has no tiles; it still takes part in the
  // merge with an empty partial.
  const int hi = min(lo + chunk, pmax + 1);
  const int ntiles = hi > lo ? (hi - lo + kTile - 1) / kTile : 0;
  const int nmt = (nqv + 15) >> 4;
  int committed = 0;                                // cp.async groups so far: one per tile, in tile order
  if (early) {
    committed = nb;
    // every row the queries can see in the early tiles must have been loaded
    if (tid == 0 && ntiles > 0 && min(hi, lo + nb * kTile) > fresh_hi && a.err)
      atomicOr(a.err, static_cast<unsigned>(ERR_RANGE));
  } else {
    for (; committed < min(nb, ntiles); ++committed) {
      issue_rows(committed, lo, INT_MAX, hi);
      cp_async_commit();
    }
  }

  const float scale = rsqrtf(static_cast<float>(HD));
  const int srow = tid >> 2, squart = tid & 3;  // softmax: query row, quarter of the tile
  float m_run = -INFINITY, l_run = 0.f;
  float acc[4][NT][4];
#pragma unroll
  for (int mt = 0; mt < 4; ++mt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.f;

  // nb tiles in flight: tiles 0 .. nb-1 now, tile i+nb-1 at the top of iteration i >= 1 (into the
  // slot of tile i-1)
  for (int i = 0; i < ntiles; ++i) {
    cp_async_wait_n(committed - (i + 1));
    __syncthreads();  // tile i visible to all; every warp is past tile i-1, so its slot is free
    if (i >= 1 && i + nb - 1 < ntiles) {
      issue_rows(i + nb - 1, lo, INT_MAX, hi);
      cp_async_commit();
      ++committed;
    }
    const int t0 = lo + i * kTile;
    const bf16* sK = reinterpret_cast<const bf16*>(sKV + (i % nb) * C::KV_TILE);
    const bf16* sV = sK + kTile * KS;

    // (1) S = Q K^T * scale, causal and range masks
    {
      const int n0 = warp * 8;
      uint32_t kb[HD / 16][2];
#pragma unroll
      for (int kk = 0; kk < HD / 16; kk += 2)
        ldsm_x4(smem_u32(sK + (n0 + (lane & 7)) * KS + kk * 16 + (lane >> 3) * 8), kb[kk][0], kb[kk][1],
                kb[kk + 1][0], kb[kk + 1][1]);
      const int pc = t0 + n0 + 2 * t4;
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        if (mt < nmt) {
          float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(smem_u32(sQ + (mt * 16 + (lane & 15)) * KS + kk * 16 + (lane >> 4) * 8), a0, a1, a2, a3);
            mma_bf16(c, a0, a1, a2, a3, kb[kk][0], kb[kk][1]);
          }
          const int qv = mt * 16 + g8;
          const int pa = sPos[qv], pb = sPos[qv + 8];
          float2 s_a, s_b;
          s_a.x = (pc < hi && pc <= pa) ? c[0] * scale : -INFINITY;
          s_a.y = (pc + 1 < hi && pc + 1 <= pa) ? c[1] * scale : -INFINITY;
          s_b.x = (pc < hi && pc <= pb) ? c[2] * scale : -INFINITY;
          s_b.y = (pc + 1 < hi && pc + 1 <= pb) ? c[3] * scale : -INFINITY;
          *reinterpret_cast<float2*>(sS + qv * SS + n0 + 2 * t4) = s_a;
          *reinterpret_cast<float2*>(sS + (qv + 8) * SS + n0 + 2 * t4) = s_b;
        }
      }
    }
    __syncthreads();

    // (2) online softmax: P = e^{S - m_new} (bf16), corr = e^{m_old - m_new}
    if (srow < nmt * 16) {  // whole warps: nmt * 64 threads
      const float4* sr = reinterpret_cast<const float4*>(sS + srow * SS + squart * 16);
      float v[16];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float4 f = sr[u];
        v[4 * u] = f.x; v[4 * u + 1] = f.y; v[4 * u + 2] = f.z; v[4 * u + 3] = f.w;
      }
      float mx = v[0];
#pragma unroll
      for (int u = 1; u < 16; ++u) mx = fmaxf(mx, v[u]);
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m_run, mx);
      const float m_use = m_new == -INFINITY ? 0.f : m_new;  // a row with nothing visible yet
      const float corr = __expf(m_run - m_use);
      uint32_t pk[8];
      float sum = 0.f;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(__expf(v[2 * u] - m_use), __expf(v[2 * u + 1] - m_use));
        sum += __low2float(h) + __high2float(h);
        pk[u] = *reinterpret_cast<const uint32_t*>(&h);
      }
      uint4* dst = reinterpret_cast<uint4*>(sP + srow * PS + squart * 16);
      dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
      dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      sum += __shfl_xor_sync(0xffffffffu, sum, 2);
      l_run = l_run * corr + sum;
      m_run = m_new;
      if (squart == 0) sCorr[srow] = corr;
    }
    __syncthreads();

    // (3) O = O * corr + P V over this warp's output dimensions
    {
      const int d0 = warp * 8 * NT;
      uint32_t vb[kTile / 16][NT][2];
#pragma unroll
      for (int kk = 0; kk < kTile / 16; ++kk) {
        const int row = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        if constexpr (NT == 2) {
          ldsm_x4_t(smem_u32(sV + row * KS + d0 + (lane >> 4) * 8), vb[kk][0][0], vb[kk][0][1], vb[kk][1][0], vb[kk][1][1]);
        } else {
          ldsm_x2_t(smem_u32(sV + row * KS + d0), vb[kk][0][0], vb[kk][0][1]);
        }
      }
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        if (mt < nmt) {
          const float ca = sCorr[mt * 16 + g8], cb = sCorr[mt * 16 + g8 + 8];
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            acc[mt][nt][0] *= ca; acc[mt][nt][1] *= ca;
            acc[mt][nt][2] *= cb; acc[mt][nt][3] *= cb;
          }
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(smem_u32(sP + (mt * 16 + (lane & 15)) * PS + kk * 16 + (lane >> 4) * 8), a0, a1, a2, a3);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) mma_bf16(acc[mt][nt], a0, a1, a2, a3, vb[kk][nt][0], vb[kk][nt][1]);
          }
        }
      }
    }
  }
  cp_async_wait<0>();  // early tiles the row positions turned out not to need

  const int d0 = warp * 8 * NT;
  if (NS == 1) {
    float* sMx = sCorr + kMaxQV;                    // the row data's max slot
    if (srow < nmt * 16 && squart == 0) {
      sL[srow] = l_run;
      sMx[srow] = m_run;
    }
    __syncthreads();
    if (Rf > 1) {
      // Flat mode merge: this split's unnormalised accumulators and (max, sum) per query vector go
      // to its slot; it counts itself in (self-resetting), and the group's last split combines the
      // Rf slots in split order: out = sum_s acc_s e^{m_s - M} / sum_s l_s e^{m_s - M}.
      const size_t sl = static_cast<size_t>(kvh) * a.flat + blockIdx.x;
      float* pacc = static_cast<float*>(a.flat_acc) + sl * (kMaxQV * HD);
      float2* pml = static_cast<float2*>(a.flat_ml);
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        if (mt >= nmt) break;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int qv = mt * 16 + g8 + 8 * half;
          if (qv >= nqv) continue;
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
            *reinterpret_cast<float2*>(pacc + qv * HD + d0 + nt * 8 + 2 * t4) =
                make_float2(acc[mt][nt][2 * half], acc[mt][nt][2 * half + 1]);
        }
      }
      if (tid < nqv) pml[sl * kMaxQV + tid] = make_float2(sMx[tid], sL[tid]);
      __threadfence();                              // the partial before the count
      __syncthreads();
      if (tid == 0) {
        unsigned* cnt = a.flat_cnt + static_cast<size_t>(g) * Hkv + kvh;
        sRecv = atomicInc(cnt, static_cast<unsigned>(Rf - 1)) == static_cast<unsigned>(Rf - 1) ? 1 : 0;
      }
      __syncthreads();
      if (!sRecv) return;
      __threadfence();                              // every split's partial is visible
      const size_t s0 = static_cast<size_t>(kvh) * a.flat + slot0;
      const float* acc0 = static_cast<const float*>(a.flat_acc) + s0 * (kMaxQV * HD);
      // weights w[q][qv] = e^{m_q - M} / sum_q l_q e^{m_q - M} in shared memory (over the K/V ring,
      // whose copies have all landed): the (max, sum) pairs staged in parallel, then one thread per
      // query vector
      float* sW = reinterpret_cast<float*>(sKV);                     // [kFlatMaxSplits][kMaxQV]
      float2* sML = reinterpret_cast<float2*>(sKV + kFlatMaxSplits * kMaxQV * 4);
      for (int i = tid; i < Rf * nqv; i += kThreads) {
        const int q = i / nqv, qv = i % nqv;
        sML[q * kMaxQV + qv] = __ldcg(&pml[(s0 + q) * kMaxQV + qv]);
      }
      __syncthreads();
      if (tid < nqv) {
        float M = -INFINITY;
        for (int q = 0; q < Rf; ++q) M = fmaxf(M, sML[q * kMaxQV + tid].x);
        float L = 0.f;
        for (int q = 0; q < Rf; ++q) {                               // in split order
          const float2 ml = sML[q * kMaxQV + tid];
          const float w = ml.x == -INFINITY ? 0.f : __expf(ml.x - M);
          sW[q * kMaxQV + tid] = w;
          L = fmaf(ml.y, w, L);
        }
        const float inv = 1.f / L;
        for (int q = 0; q < Rf; ++q) sW[q * kMaxQV + tid] *= inv;
      }
      __syncthreads();
      for (int e = tid; e < nqv * (HD / 4); e += kThreads) {
        const int qv = e / (HD / 4), d4 = e % (HD / 4);
        const float4* src = reinterpret_cast<const float4*>(acc0 + qv * HD) + d4;
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int q0 = 0; q0 < Rf; q0 += 8) {                        // 8 slots' loads in flight
          float4 v[8];
#pragma unroll
          for (int u = 0; u < 8; ++u)
            if (q0 + u < Rf) v[u] = __ldcg(src + static_cast<size_t>(q0 + u) * (kMaxQV * HD / 4));
#pragma unroll
          for (int u = 0; u < 8; ++u)
            if (q0 + u < Rf) {
              const float w = sW[(q0 + u) * kMaxQV + qv];
              o.x = fmaf(w, v[u].x, o.x); o.y = fmaf(w, v[u].y, o.y);
              o.z = fmaf(w, v[u].z, o.z); o.w = fmaf(w, v[u].w, o.w);
            }
        }
        const size_t rh = static_cast<size_t>(r0 + qv / G) * a.H + kvh * G + qv % G;
        *reinterpret_cast<uint2*>(static_cast<bf16*>(a.out) + rh * HD + d4 * 4) =
            make_uint2(pack_bf2(o.x, o.y), pack_bf2(o.z, o.w));
      }
      return;
    }
#pragma unroll
    for (int mt = 0; mt < 4; ++mt) {
      if (mt >= nmt) break;
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int qv = mt * 16 + g8 + 8 * half;
        if (qv >= nqv) continue;
        const size_t rh = static_cast<size_t>(r0 + qv / G) * a.H + kvh * G + qv % G;
        const float inv = 1.f / sL[qv];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          *reinterpret_cast<__nv_bfloat162*>(static_cast<bf16*>(a.out) + rh * HD + d0 + nt * 8 + 2 * t4) =
              __floats2bfloat162_rn(acc[mt][nt][2 * half] * inv, acc[mt][nt][2 * half + 1] * inv);
      }
    }
    return;
  }

  // Split merge: out = sum_s acc_s e^{m_s - M} / sum_s l_s e^{m_s - M}, M = max_s m_s. Element e
  // of the group (query vector e / (hd/4), dimensions 4 (e % (hd/4)) ..) belongs to the split r
  // with r E4 / NS <= e < (r+1) E4 / NS. Splits that hold no position a row can see contribute
  // m = -inf, l = 0, acc = 0, hence weight 0.
  if (ring) {                                       // the receive buffers lie over this CTA's ring
    __syncthreads();                                // every warp is past its last K/V read
    cluster_arrive_release();
  }
  cluster_wait();                                   // every split's receive barrier is armed (and ring free)
  if (srow < nqv && squart == 0) {                  // (max, sum) of the query vector to every split
    const uint32_t src = smem_u32(rML + rank * QR + srow);
    for (int s2 = 0; s2 < NS; ++s2)
      st_async_v2(dsmem_addr(src, static_cast<uint32_t>(s2)), dsmem_addr(rbar, static_cast<uint32_t>(s2)), m_run,
                  l_run);
  }
#pragma unroll
  for (int mt = 0; mt < 4; ++mt) {
    if (mt >= nmt) break;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int qv = mt * 16 + g8 + 8 * half;
      if (qv >= nqv) continue;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int d = d0 + nt * 8 + 2 * t4;
        const int e = qv * (HD / 4) + (d >> 2);
        const int owner = ((e + 1) * NS - 1) / E4;
        const uint32_t dst = smem_u32(rAcc + rank * share + (e - owner * E4 / NS)) + static_cast<uint32_t>((d & 3) * 4);
        st_async_v2(dsmem_addr(dst, static_cast<uint32_t>(owner)), dsmem_addr(rbar, static_cast<uint32_t>(owner)),
                    acc[mt][nt][2 * half], acc[mt][nt][2 * half + 1]);
      }
    }
  }
  if (tid == 0) {
    sRecv = tc::wait_bar_budget(rbar, 0, tc::kWaitCycles) ? 1 : 0;
    if (!sRecv) {
      if (a.err) atomicOr(a.err, static_cast<unsigned>(ERR_TIMEOUT));
      tc::wait_bar_budget(rbar, 0, tc::kDrainCycles);   // let partials still in flight land before leaving
    }
  }
  __syncthreads();
  if (!sRecv) return;
  if (R > 1) {
    ctx_cluster_merge<HD>(a, rML, rAcc, QR, share, e_lo, e_hi, g, kvh, rank, cr, R, r0, G, &sRecv);
    return;
  }
  for (int e = e_lo + tid; e < e_hi; e += kThreads) {
    const int qv = e / (HD / 4), d4 = e % (HD / 4);
    // every split's values are loaded first (indices clamped, so no load waits behind a branch),
    // then combined in split order; splits past NS are selected away
    float2 ml[kMaxSplits];
#pragma unroll
    for (int s2 = 0; s2 < kMaxSplits; ++s2) ml[s2] = rML[min(s2, NS - 1) * QR + qv];
    float M = -INFINITY;
#pragma unroll
    for (int s2 = 0; s2 < kMaxSplits; ++s2) M = s2 < NS ? fmaxf(M, ml[s2].x) : M;
    float w[kMaxSplits];
    float Lsum = 0.f;
#pragma unroll
    for (int s2 = 0; s2 < kMaxSplits; ++s2) {
      w[s2] = __expf(ml[s2].x - M);
      Lsum = s2 < NS ? Lsum + ml[s2].y * w[s2] : Lsum;
    }
    const float inv = 1.f / Lsum;
    float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int s2 = 0; s2 < kMaxSplits; ++s2) {
      const float ws = w[s2] * inv;
      const float4 v = rAcc[min(s2, NS - 1) * share + (e - e_lo)];
      if (s2 < NS) {
        o.x = fmaf(ws, v.x, o.x); o.y = fmaf(ws, v.y, o.y);
        o.z = fmaf(ws, v.z, o.z); o.w = fmaf(ws, v.w, o.w);
      }
    }
    const size_t rh = static_cast<size_t>(r0 + qv / G) * a.H + kvh * G + qv % G;
    *reinterpret_cast<uint2*>(static_cast<bf16*>(a.out) + rh * HD + d4 * 4) =
        make_uint2(pack_bf2(o.x, o.y), pack_bf2(o.z, o.w));
  }
}

// Dynamic shared memory each of n resident CTAs can take: the SM's capacity split n ways, less the
// per-block reservation and the kernel's static arrays (with a little room).
size_t smem_share(int n) {
  static const int sm_bytes = [] {
    int dev = 0, v = 0;
    cudaGetDevice(&dev);
    return cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) == cudaSuccess ? v : 0;
  }();
  static const int reserved = [] {
    int dev = 0, v = 0;
    cudaGetDevice(&dev);
    return cudaDeviceGetAttribute(&v, cudaDevAttrReservedSharedMemoryPerBlock, dev) == cudaSuccess ? v : 1024;
  }();
  const long share = static_cast<long>(sm_bytes) / n - reserved - 256;
  return share > 0 ? static_cast<size_t>(share) : 0;
}

template <int HD, int DEC>
cudaError_t configure() {
  static cudaError_t e = [] {
    cudaError_t r = cudaFuncSetAttribute(attn_kernel<HD, DEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
    if (r == cudaSuccess)
      r = cudaFuncSetAttribute(attn_kernel<HD, DEC>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return r;
  }();
  return e;
}

// Whether clusters of n CTAs of the largest step-shape attention CTA can be scheduled.
template <int HD>
bool clusters_fit(int n) {
  if (configure<HD, 0>() != cudaSuccess) return false;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(n, 1, 1);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = AttnCfg<HD>::bytes(kMaxQV, 2 * kTile, n, 2, 0);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(n);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  return cudaOccupancyMaxActiveClusters(&clusters, attn_kernel<HD, 0>, &cfg) == cudaSuccess && clusters > 0;
}

// The launch's K/V ring and shared memory: the deepest ring (2 to 4 tiles, at most the chunk's)
// within the shared memory a CTA may take, its share of the SM when the grid needs several CTAs
// per SM resident (up to the register bound), the opt-in maximum otherwise. The merge buffers go
// over the ring only where that is what makes it fit.
struct Shape {
  int nb, ring;
  size_t smem;
  bool dec;      // the decode instantiation (one context cluster, separate merge buffers)
};

template <int HD>
Shape shape_of(const AttnArgs& a) {
  using C = AttnCfg<HD>;
  const int qr = C::qrows(a.max_rows, a.H / a.kv.Hkv), ns = a.n_splits;
  const int max_nb = a.chunk > kTile ? std::min(kMaxBuf, a.chunk / kTile) : 1;
  const int R = a.n_ctx_clusters > 1 ? a.n_ctx_clusters : 1;
  const long ctas = a.flat > 0 ? static_cast<long>(a.flat) * a.kv.Hkv : static_cast<long>(ns) * R * a.n_groups * a.kv.Hkv;
  const long sms = sm_count_cached();
  const int per_sm = static_cast<int>(std::min<long>(kCtasPerSm<HD>, (ctas + sms - 1) / sms));
  const size_t cap = per_sm <= 1 ? static_cast<size_t>(kMaxSmem) : smem_share(per_sm);
  Shape sh{std::min(2, max_nb), 0, 0, false};
  bool found = false;
  for (int n = max_nb; n >= std::min(2, max_nb) && !found; --n)
    for (int r = 0; r <= 1 && !found; ++r) {
      if (r && (ns == 1 || C::merge_bytes(qr, ns) > static_cast<size_t>(n) * C::KV_TILE)) continue;
      if (C::bytes(qr, a.chunk, ns, n, r) <= cap) {
        sh.nb = n;
        sh.ring = r;
        found = true;
      }
    }
  sh.smem = C::bytes(qr, a.chunk, ns, sh.nb, sh.ring);
  sh.dec = a.pre_len && R == 1 && !sh.ring && a.flat <= 0;
  return sh;
}

template <int HD>
cudaError_t launch(const AttnArgs& a, cudaStream_t st) {
  const cudaError_t e = configure<HD, 0>();
  if (e != cudaSuccess) return e;
  const cudaError_t e1 = configure<HD, 1>();
  if (e1 != cudaSuccess) return e1;
  const Shape sh = shape_of<HD>(a);
  if (sh.smem > static_cast<size_t>(kMaxSmem)) return cudaErrorInvalidValue;
  const int ns = a.n_splits, R = a.n_ctx_clusters > 1 ? a.n_ctx_clusters : 1;
  const dim3 grid = a.flat > 0 ? dim3(a.flat, 1, a.kv.Hkv) : dim3(ns * R, a.n_groups, a.kv.Hkv);
  if (sh.dec)
    return launch_pdl_cluster(attn_kernel<HD, 1>, grid, dim3(kThreads), sh.smem, st, ns, a, sh.nb, sh.ring);
  return launch_pdl_cluster(attn_kernel<HD, 0>, grid, dim3(kThreads), sh.smem, st, ns, a, sh.nb, sh.ring);
}

// Clusters of this shape the device holds at once (cudaOccupancyMaxActiveClusters, remembered per
// instantiation, cluster size and shared memory: the answer depends on how clusters pack into the
// GPCs, which a per-SM count does not see).
template <int HD>
int max_clusters(const Shape& sh, int ns) {
  static std::mutex mu;
  static std::vector<std::array<long, 3>> seen;   // (dec * 32 + ns, smem, clusters)
  const long key = (sh.dec ? 32 : 0) + ns;
  {
    std::lock_guard<std::mutex> lk(mu);
    for (const auto& v : seen)
      if (v[0] == key && v[1] == static_cast<long>(sh.smem)) return static_cast<int>(v[2]);
  }
  if (configure<HD, 0>() != cudaSuccess || configure<HD, 1>() != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(ns, 1, 1);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = sh.smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(ns);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  const cudaError_t e = sh.dec ? cudaOccupancyMaxActiveClusters(&n, attn_kernel<HD, 1>, &cfg)
                               : cudaOccupancyMaxActiveClusters(&n, attn_kernel<HD, 0>, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  std::lock_guard<std::mutex> lk(mu);
  seen.push_back({key, static_cast<long>(sh.smem), static_cast<long>(n)});
  return n;
}

template <int HD>
int clusters_max(const AttnArgs& a) {
  const Shape sh = shape_of<HD>(a);
  if (sh.smem > static_cast<size_t>(kMaxSmem)) return 0;
  return max_clusters<HD>(sh, a.n_splits);
}

}  // namespace

int attention_ctas_per_sm(int hd) { return hd == 64 ? kCtasPerSm<64> : kCtasPerSm<128>; }

int attention_max_splits() {
  static const int n = (clusters_fit<128>(kMaxSplits) && clusters_fit<64>(kMaxSplits)) ? kMaxSplits : 8;
  return n;
}

int attention_max_clusters(const AttnArgs& a) {
  if (a.n_splits < 1 || a.n_splits > kMaxSplits || a.chunk <= 0 || a.kv.Hkv <= 0 || a.H % a.kv.Hkv != 0) return 0;
  if (a.hd == 128) return clusters_max<128>(a);
  if (a.hd == 64) return clusters_max<64>(a);
  return 0;
}

cudaError_t attention(const AttnArgs& a, cudaStream_t st) {
  if (a.n_groups <= 0) return cudaSuccess;
  if (a.n_splits < 1 || a.n_splits > kMaxSplits || a.chunk <= 0 || a.chunk % kTile != 0) return cudaErrorInvalidValue;
  if (a.kv.Hkv <= 0 || a.H % a.kv.Hkv != 0 || a.max_rows < 1 || a.max_rows * (a.H / a.kv.Hkv) > kMaxQV)
    return cudaErrorInvalidValue;
  if (a.n_ctx_clusters > 1 && (a.n_splits < 2 || !a.part_acc || !a.part_ml || !a.part_cnt)) return cudaErrorInvalidValue;
  if (a.flat > 0 && (!a.pre_len || a.n_splits != 1 || a.n_ctx_clusters > 1 || a.n_groups > a.flat || a.n_groups > 64 ||
                     a.chunk < 2 * kTile ||   // a ring of two tiles holds the merge's weights
                     !a.flat_acc || !a.flat_ml || !a.flat_cnt))
    return cudaErrorInvalidValue;
  if (a.hd == 128) return launch<128>(a, st);
  if (a.hd == 64) return launch<64>(a, st);
  return cudaErrorInvalidValue;
}

}  // namespace sd2
