// Persistent decoder-layer chain: every layer of one forward pass over at most 16 token rows (a
// drafter step of Sec. 3.2, Eq. 2 steering included) in one cooperative launch, one CTA per SM.
//
// Per layer the pass runs five phases separated by grid-wide barriers:
//   Q  q,k,v projections          x_l -> split-K partials Pq
//   A  attention                  sum Pq, rotary, new K/V into the paged cache, one 64-position
//                                 tile per (split, row group, KV head) unit -> partials Pa
//   O  output projection          merged Pa -> split-K partials Po
//   U  gate/up projections + Eq.2 RMSNorm(x_l + sum Po) -> h = (W_u a + b) * SiLU(W_g a)
//   D  down projection            h -> split-K partials Pd;  x_{l+1} = x_l + sum Po + sum Pd
// Each phase builds its GEMM operand itself from what the previous phases left in L2 (sums of
// partials, the RMSNorm row scale, the attention merge), so no phase needs a separate reduction
// pass. The weights never wait for a barrier: warp 0 streams the weight tiles of all of this CTA's
// units of all layers, in order, through one TMA ring, so HBM keeps streaming while the CTAs meet
// at a barrier; warp 1 issues tcgen05.mma into TMEM; warps 2-5 build operands, read accumulators
// back, run the epilogues and the attention. Every wait is bounded: on expiry the kernel records
// ERR_TIMEOUT, stops all roles and frees TMEM.
#include <cuda.h>
#include <math.h>

#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "sd2.h"
#include "tc.cuh"

namespace sd2 {
namespace {

using namespace tc;

constexpr int kThreads = 192;
constexpr int kW = 128;                  // weight rows per tile (MMA M)
constexpr int kBK = 64;                  // K per k-block (128 bytes of bf16)
constexpr int kNT = 16;                  // token columns (MMA N)
constexpr int kAStage = kW * kBK * 2;    // one weight tile: 16 KB
constexpr int kBBlock = kNT * kBK * 2;   // one token k-block: 2 KB
constexpr int kBRegion = 64 * 1024;      // token operand of up to 32 k-blocks; attention overlays it
constexpr int kSmem = 227 * 1024;
constexpr int kMaps = 7;                 // per layer: q, k, v, o, gate, up, down
constexpr int kQV = 16;                  // attention query vectors per unit (one m-tile)
constexpr int kTileP = 64;               // attention positions per tile

struct ChainK {
  const CUtensorMap* maps;               // [L][kMaps]
  const bf16* const* norms;              // [L][2]: attention norm, MLP norm
  const bf16* embed;
  int L, d, H, Hkv, hd, F, vocab;
  float eps;
  int M;
  const int *tok, *row_pos, *row_seq, *row_valid;
  const int *grp_row0, *grp_nrows, *grp_seq;
  int n_groups, n_splits, chunk;
  KVCache kv;
  const float* rope_cs;
  const float* bias;
  int ld_bias;
  float* x_out;
  float *xbuf, *pq, *po, *pd, *pa;
  bf16* h;
  unsigned* sync;
  unsigned* err;
  int n_cta, sp_q, sp_o, sp_d, stages;
};

// ------------------------------------------------------------------------------ work split
// GEMM phases of one layer: tiles of 128 weight rows (SwiGLU: 64 gate + 64 up rows), K in 64-wide
// blocks split over sp CTAs. Unit u of a phase: tile u / sp, K slice u % sp.
struct Gemm {
  int tiles, sp, kb;                     // weight tiles, K slices, K blocks
};
__device__ __forceinline__ Gemm gemm_of(const ChainK& a, int ph) {
  const int nq = (a.H + 2 * a.Hkv) * a.hd;
  if (ph == 0) return {nq / kW, a.sp_q, a.d / kBK};
  if (ph == 1) return {a.d / kW, a.sp_o, a.H * a.hd / kBK};
  if (ph == 2) return {a.F / 64, 1, a.d / kBK};
  return {a.d / kW, a.sp_d, a.F / kBK};
}
__device__ __forceinline__ int kb_lo(const Gemm& g, int slice) { return slice * g.kb / g.sp; }

// ------------------------------------------------------------------------------ grid barrier
__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// All CTAs' workers: arrive at barrier number `b`, then wait until every CTA has. Worker thread 0
// does the global part; the named barriers order the other workers' memory operations around it.
__device__ __forceinline__ bool grid_sync(const ChainK& a, unsigned b, volatile int* abort_flag, int* ok_shared) {
  asm volatile("bar.sync 1, 128;" ::: "memory");
  if (threadIdx.x == 64) {
    int ok = *abort_flag == 0;
    if (ok) {
      __threadfence();
      atomicAdd(a.sync, 1u);
      const unsigned target = static_cast<unsigned>(a.n_cta) * (b + 1);
      const long long t0 = clock64();
      while (ld_acquire(a.sync) < target) {
        if (*abort_flag) { ok = 0; break; }
        if (clock64() - t0 > kWaitCycles) {
          *abort_flag = 1;
          atomicOr(a.err, static_cast<unsigned>(ERR_TIMEOUT));
          ok = 0;
          break;
        }
      }
    }
    *ok_shared = ok;
  }
  asm volatile("bar.sync 1, 128;" ::: "memory");
  return *ok_shared != 0;
}

// ------------------------------------------------------------------------------ operand helpers
// byte offset of 16-byte chunk c (0..7) of token row m in a 128-byte-swizzled k-block
__device__ __forceinline__ uint32_t sw_off(int m, int c) { return static_cast<uint32_t>(m * 128 + ((c ^ (m & 7)) << 4)); }
__device__ __forceinline__ uint32_t pack2(float x, float y) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ float block_sum128(float v, float* red) {
  v = warp_sum(v);
  const int w = (threadIdx.x - 64) >> 5, l = threadIdx.x & 31;
  asm volatile("bar.sync 1, 128;" ::: "memory");
  if (l == 0) red[w] = v;
  asm volatile("bar.sync 1, 128;" ::: "memory");
  const float s = red[0] + red[1] + red[2] + red[3];
  asm volatile("bar.sync 1, 128;" ::: "memory");
  return s;
}

// v += sum over slices s < n of p[s * stride + 0..7] (and w += the same at q), in slice order.
// The loads of four slices are issued before any of them is added, so a thread waits for one
// L2 round trip per four slices instead of one per slice. All of these buffers are written by
// other CTAs earlier in this launch: they are read from L2, never from a stale L1 line.
__device__ __forceinline__ void add8(float (&v)[8], const float4& x, const float4& y) {
  v[0] += x.x; v[1] += x.y; v[2] += x.z; v[3] += x.w; v[4] += y.x; v[5] += y.y; v[6] += y.z; v[7] += y.w;
}
__device__ __forceinline__ void add_slices(const float* p, const float* q, size_t stride, int n, float (&v)[8],
                                           float (&w)[8], bool two) {
  const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s0 = 0; s0 < n; s0 += 4) {
    float4 t[4][4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      t[u][0] = t[u][1] = t[u][2] = t[u][3] = z;
      if (s0 + u < n) {
        const size_t o = static_cast<size_t>(s0 + u) * stride;
        t[u][0] = __ldcg(reinterpret_cast<const float4*>(p + o));
        t[u][1] = __ldcg(reinterpret_cast<const float4*>(p + o + 4));
        if (two) {
          t[u][2] = __ldcg(reinterpret_cast<const float4*>(q + o));
          t[u][3] = __ldcg(reinterpret_cast<const float4*>(q + o + 4));
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      add8(v, t[u][0], t[u][1]);
      add8(w, t[u][2], t[u][3]);
    }
  }
}
// Residual stream rows: buffer 0 holds x_l (the input of layer l), buffer 1 holds x'_l = x_l + the
// attention output of layer l (the input of its MLP). Each is written by its owner CTAs in the
// phase that first needs it and read by everyone from the next phase on.
__device__ __forceinline__ float* xrow(const ChainK& a, int buf, int m) {
  return a.xbuf + (static_cast<size_t>(buf) * kNT + m) * a.d;
}
// 8 columns at c and at c2 (two = both) of base[m] + sum over the n slices of P[s][m]
__device__ __forceinline__ void row_plus_slices(const ChainK& a, const float* base, const float* P, int n, int m,
                                                int c, int c2, bool two, float (&v)[8], float (&w)[8]) {
  const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  float4 b0 = __ldcg(reinterpret_cast<const float4*>(base + c)), b1 = __ldcg(reinterpret_cast<const float4*>(base + c + 4));
  float4 b2 = z, b3 = z;
  if (two) {
    b2 = __ldcg(reinterpret_cast<const float4*>(base + c2));
    b3 = __ldcg(reinterpret_cast<const float4*>(base + c2 + 4));
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) { v[i] = 0.f; w[i] = 0.f; }
  add8(v, b0, b1);
  add8(w, b2, b3);
  const float* p = P + static_cast<size_t>(m) * a.d;
  add_slices(p + c, p + c2, static_cast<size_t>(kNT) * a.d, n, v, w, two);
}

// ------------------------------------------------------------------------------ the kernel
__global__ void __launch_bounds__(kThreads, 1) chain_kernel(const __grid_constant__ ChainK a) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = a.stages;
  unsigned char* ring = smem;
  unsigned char* breg = smem + static_cast<size_t>(S) * kAStage;          // token operand / attention
  uint64_t* bars = reinterpret_cast<uint64_t*>(breg + kBRegion);          // full[S], empty[S], bready, tfull, tempty
  float* xch = reinterpret_cast<float*>(bars + 2 * S + 4);                 // [64][17] SwiGLU exchange
  float* red = xch + 64 * 17;                                              // [8] reductions
  float* rsd = red + 8;                                                    // [16] row scales
  float* wts = rsd + 16;                                                   // [16][32][2] merge weights
  volatile int* flags = reinterpret_cast<volatile int*>(wts + 16 * 32 * 2);   // [0] abort [1] tmem [2] ok
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, bready = empty0 + 8 * S, tfull = bready + 8,
                 tempty = tfull + 8;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cta = blockIdx.x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(bready, 1);
    mbar_init(tfull, 1);
    mbar_init(tempty, 1);
    flags[0] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<int*>(flags) + 1), 32);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = static_cast<uint32_t>(flags[1]);
  volatile int* abort_flag = flags;

  if (warp == 0) {
    // ---------------------------------------------------------------- weight stream (TMA)
    if (lane == 0) {
      const uint64_t pol = l2_evict_first();
      uint32_t j = 0;
      bool ok = true;
      for (int l = 0; l < a.L && ok; ++l) {
        const CUtensorMap* mp = a.maps + static_cast<size_t>(l) * kMaps;
        for (int ph = 0; ph < 4 && ok; ++ph) {
          const Gemm g = gemm_of(a, ph);
          for (int u = cta; u < g.tiles * g.sp && ok; u += a.n_cta) {
            const int t = u / g.sp, sl = u % g.sp;
            for (int kb = kb_lo(g, sl); kb < kb_lo(g, sl + 1); ++kb, ++j) {
              const uint32_t s = j % S;
              if (j >= static_cast<uint32_t>(S) && !wait_bar(empty0 + 8 * s, ((j / S) & 1) ^ 1, abort_flag, a.err)) {
                ok = false;
                break;
              }
              mbar_expect_tx(full0 + 8 * s, kAStage);
              const uint32_t dst = smem_u32(ring + static_cast<size_t>(s) * kAStage);
              if (ph == 0) {
                int row = t * kW, m = 0;
                const int rq = a.H * a.hd, rk = a.Hkv * a.hd;
                if (row >= rq) { row -= rq; m = 1; if (row >= rk) { row -= rk; m = 2; } }
                tma_load_2d_stream(dst, mp + m, kb * kBK, row, full0 + 8 * s, pol);
              } else if (ph == 1) {
                tma_load_2d_stream(dst, mp + 3, kb * kBK, t * kW, full0 + 8 * s, pol);
              } else if (ph == 2) {
                tma_load_2d_stream(dst, mp + 4, kb * kBK, t * 64, full0 + 8 * s, pol);
                tma_load_2d_stream(dst + kAStage / 2, mp + 5, kb * kBK, t * 64, full0 + 8 * s, pol);
              } else {
                tma_load_2d_stream(dst, mp + 6, kb * kBK, t * kW, full0 + 8 * s, pol);
              }
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issue (one thread)
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kW, kNT);
      uint32_t j = 0, nb = 0;
      bool ok = true;
      for (int l = 0; l < a.L && ok; ++l) {
        for (int ph = 0; ph < 4 && ok; ++ph) {
          const Gemm g = gemm_of(a, ph);
          for (int u = cta; u < g.tiles * g.sp && ok; u += a.n_cta, ++nb) {
            const int sl = u % g.sp;
            if (!wait_bar(bready, nb & 1, abort_flag, a.err)) { ok = false; break; }
            if (nb > 0 && !wait_bar(tempty, (nb - 1) & 1, abort_flag, a.err)) { ok = false; break; }
            tc_fence_after();
            const int k0 = kb_lo(g, sl), k1 = kb_lo(g, sl + 1);
            for (int kb = k0; kb < k1; ++kb, ++j) {
              const uint32_t s = j % S;
              if (!wait_bar(full0 + 8 * s, (j / S) & 1, abort_flag, a.err)) { ok = false; break; }
              tc_fence_after();
              const uint64_t ad = sw128_desc(smem_u32(ring + static_cast<size_t>(s) * kAStage));
              const uint64_t bd = sw128_desc(smem_u32(breg + static_cast<size_t>(kb - k0) * kBBlock));
#pragma unroll
              for (int kk = 0; kk < kBK / 16; ++kk)
                mma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb > k0 || kk > 0) ? 1u : 0u);
              mma_commit(empty0 + 8 * s);
            }
            if (ok) mma_commit(tfull);
          }
        }
      }
    }
  } else {
    // ---------------------------------------------------------------- workers (warps 2-5)
    const int tid = threadIdx.x - 64;
    const int q = warp & 3, r = q * 32 + lane;           // TMEM lane quarter, weight row of the tile
    int* ok_shared = const_cast<int*>(flags) + 2;
    const int M = a.M;
    const int nq = (a.H + 2 * a.Hkv) * a.hd;
    const int G = a.H / a.Hkv, half = a.hd / 2;
    uint32_t nb = 0;                                       // GEMM units done by this CTA
    unsigned bar_no = 0;
    bool ok = true;
    // owned columns of the residual stream (written once per layer)
    const int own_lo = (cta * (a.d / 8) / a.n_cta) * 8, own_hi = ((cta + 1) * (a.d / 8) / a.n_cta) * 8;

    // Epilogue of a Q/O/D unit: this tile's K-slice partial, P[slice][m][tile rows] for m < M.
    auto store_partial = [&](float* P, int ncols, int t, int sl) {
      if (!wait_bar(tfull, nb & 1, abort_flag, a.err)) { ok = false; return; }
      tc_fence_after();
      float v[16];
      tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16), v);
#pragma unroll
      for (int m = 0; m < kNT; ++m)
        if (m < M) P[(static_cast<size_t>(sl) * kNT + m) * ncols + t * kW + r] = v[m];
      tc_fence_before();
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (tid == 0) mbar_arrive(tempty);
    };
    // Token operand ready for the MMA thread (generic-proxy writes -> tensor-core reads).
    auto b_ready = [&]() {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (tid == 0) mbar_arrive(bready);
    };

    // Token row m of an RMSNorm'd GEMM operand: x = base[m] + sum of the n slices P[s][m] (base null:
    // the embedding of the row's token), over all d columns (thread: column groups tid, tid + 128);
    // the owned columns of x go to residual buffer `dst`; with `build`, k-blocks k0..k1 of the
    // operand get bf16(x * rsqrt(mean(x^2) + eps) * gamma).
    auto norm_build = [&](int m, const float* base, const float* P, int n, int dst, const bf16* gamma, bool build,
                          int k0, int k1) {
      const int c0 = tid * 8, c1 = (tid + 128) * 8;
      const bool has0 = c0 < a.d, has1 = c1 < a.d;
      float x0[8], x1[8];
      if (!base) {
        const int t = min(max(a.tok[m], 0), a.vocab - 1);
        const bf16* er = a.embed + static_cast<size_t>(t) * a.d;
        uint4 e0 = make_uint4(0, 0, 0, 0), e1 = e0;
        if (has0) e0 = *reinterpret_cast<const uint4*>(er + c0);
        if (has1) e1 = *reinterpret_cast<const uint4*>(er + c1);
        x0[0] = bf_lo(e0.x); x0[1] = bf_hi(e0.x); x0[2] = bf_lo(e0.y); x0[3] = bf_hi(e0.y);
        x0[4] = bf_lo(e0.z); x0[5] = bf_hi(e0.z); x0[6] = bf_lo(e0.w); x0[7] = bf_hi(e0.w);
        x1[0] = bf_lo(e1.x); x1[1] = bf_hi(e1.x); x1[2] = bf_lo(e1.y); x1[3] = bf_hi(e1.y);
        x1[4] = bf_lo(e1.z); x1[5] = bf_hi(e1.z); x1[6] = bf_lo(e1.w); x1[7] = bf_hi(e1.w);
      } else if (has0) {
        row_plus_slices(a, base, P, n, m, c0, c1, has1, x0, x1);
      }
      float ss = 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) ss += (has0 ? x0[i] * x0[i] : 0.f) + (has1 ? x1[i] * x1[i] : 0.f);
      float* xd = xrow(a, dst, m);
      if (has0 && c0 >= own_lo && c0 < own_hi) {
        *reinterpret_cast<float4*>(xd + c0) = make_float4(x0[0], x0[1], x0[2], x0[3]);
        *reinterpret_cast<float4*>(xd + c0 + 4) = make_float4(x0[4], x0[5], x0[6], x0[7]);
      }
      if (has1 && c1 >= own_lo && c1 < own_hi) {
        *reinterpret_cast<float4*>(xd + c1) = make_float4(x1[0], x1[1], x1[2], x1[3]);
        *reinterpret_cast<float4*>(xd + c1 + 4) = make_float4(x1[4], x1[5], x1[6], x1[7]);
      }
      ss = block_sum128(ss, red);
      if (!build) return;
      const float rs = rsqrtf(ss / static_cast<float>(a.d) + a.eps);
#pragma unroll
      for (int gi = 0; gi < 2; ++gi) {
        const int c8 = tid + gi * 128;
        if (c8 * 8 >= a.d) continue;
        const int kb = c8 >> 3;
        if (kb < k0 || kb >= k1) continue;
        const float* xv = gi ? x1 : x0;
        const uint4 gm = *reinterpret_cast<const uint4*>(gamma + c8 * 8);
        const uint4 o = make_uint4(pack2(xv[0] * rs * bf_lo(gm.x), xv[1] * rs * bf_hi(gm.x)),
                                   pack2(xv[2] * rs * bf_lo(gm.y), xv[3] * rs * bf_hi(gm.y)),
                                   pack2(xv[4] * rs * bf_lo(gm.z), xv[5] * rs * bf_hi(gm.z)),
                                   pack2(xv[6] * rs * bf_lo(gm.w), xv[7] * rs * bf_hi(gm.w)));
        *reinterpret_cast<uint4*>(breg + (kb - k0) * kBBlock + sw_off(m, c8 & 7)) = o;
      }
    };

    for (int l = 0; l < a.L && ok; ++l) {
      const bf16* g_attn = a.norms[2 * l];
      const bf16* g_mlp = a.norms[2 * l + 1];
      // ============================================================ Q: x_l -> Pq
      if (l > 0 && !(ok = grid_sync(a, bar_no++, abort_flag, ok_shared))) break;
      {
        const Gemm g = gemm_of(a, 0);
        const bool has = cta < g.tiles * g.sp;
        const int sl = cta % g.sp, k0 = kb_lo(g, sl), k1 = kb_lo(g, sl + 1);
        for (int m = 0; m < kNT; ++m) {
          if (m >= M) {      // zero token rows beyond M
            if (has)
              for (int cc = tid; cc < (k1 - k0) * 8; cc += 128)
                *reinterpret_cast<uint4*>(breg + (cc >> 3) * kBBlock + sw_off(m, cc & 7)) = make_uint4(0, 0, 0, 0);
            continue;
          }
          if (l == 0) {
            norm_build(m, nullptr, nullptr, 0, 0, g_attn, has, k0, k1);
          } else {
            norm_build(m, xrow(a, 1, m), a.pd, a.sp_d, 0, g_attn, has, k0, k1);
          }
        }
        if (has) {
          b_ready();
          store_partial(a.pq, nq, cta / g.sp, sl);
          ++nb;
        }
      }
      if (!ok || !(ok = grid_sync(a, bar_no++, abort_flag, ok_shared))) break;

      // ============================================================ A: attention units
      {
        const int KS = a.hd + 8, SS = kTileP + 8, PS = kTileP + 8;
        bf16* sQ = reinterpret_cast<bf16*>(breg);                              // [16][KS]
        bf16* sK = sQ + kQV * KS;                                              // [64][KS]
        bf16* sV = sK + kTileP * KS;                                           // [64][KS]
        float* sS = reinterpret_cast<float*>(sV + kTileP * KS);                // [16][SS]
        bf16* sP = reinterpret_cast<bf16*>(sS + kQV * SS);                     // [16][PS]
        float* sCorr = reinterpret_cast<float*>(sP + kQV * PS);                // [16]
        int* sPos = reinterpret_cast<int*>(sCorr + kQV);                       // [16]
        const int n_units = a.n_splits * a.n_groups * a.Hkv;
        const int g8 = lane >> 2, t4 = lane & 3, w4 = tid >> 5;
        const bf16* pool = static_cast<const bf16*>(a.kv.pool);
        bf16* poolw = static_cast<bf16*>(a.kv.pool);
        const size_t head_stride = static_cast<size_t>(16) * a.hd;
        const size_t blk_stride = static_cast<size_t>(2) * a.Hkv * head_stride;
        for (int u = cta; u < n_units; u += a.n_cta) {
          const int split = u % a.n_splits, rest = u / a.n_splits;
          const int gi = rest % a.n_groups, kvh = rest / a.n_groups;
          const int r0 = a.grp_row0[gi], nr = a.grp_nrows[gi], seq = a.grp_seq[gi];
          const int nqv = nr * G;
          int pmax = 0;
          for (int i = 0; i < nr; ++i) pmax = max(pmax, a.row_pos[r0 + i]);
          const int lo = split * a.chunk;
          const int hi = min(lo + a.chunk, pmax + 1);
          const float2* cs = reinterpret_cast<const float2*>(a.rope_cs);
          // queries: sum the K-slice partials, rotate (rotate-half pairs), bf16
          for (int e = tid; e < kQV * half; e += 128) {
            const int qv = e / half, i = e % half;
            float x1 = 0.f, x2 = 0.f;
            if (qv < nqv) {
              const int m = r0 + qv / G, hh = kvh * G + qv % G;
              const float* p = a.pq + static_cast<size_t>(m) * nq + hh * a.hd + i;
              for (int s0 = 0; s0 < a.sp_q; s0 += 4) {     // four slices' loads in flight at once
                float t1[4], t2[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                  const bool in = s0 + u < a.sp_q;
                  const float* pp = p + static_cast<size_t>(in ? s0 + u : 0) * kNT * nq;
                  t1[u] = in ? __ldcg(pp) : 0.f;
                  t2[u] = in ? __ldcg(pp + half) : 0.f;
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) { x1 += t1[u]; x2 += t2[u]; }
              }
              const float2 c = cs[static_cast<size_t>(a.row_pos[m]) * half + i];
              const float o1 = x1 * c.x - x2 * c.y, o2 = x2 * c.x + x1 * c.y;
              x1 = o1; x2 = o2;
            }
            sQ[qv * KS + i] = __float2bfloat16_rn(x1);
            sQ[qv * KS + i + half] = __float2bfloat16_rn(x2);
          }
          if (tid < kQV) sPos[tid] = tid < nqv ? a.row_pos[r0 + tid / G] : -1;
          // new rows of this split: K (rotated) and V into the paged cache
          for (int e = tid; e < nr * half; e += 128) {
            const int rr = e / half, i = e % half, m = r0 + rr;
            const int pos = a.row_pos[m];
            if (pos < lo || pos >= lo + a.chunk || !a.row_valid[m]) continue;
            float k1 = 0.f, k2 = 0.f, v1 = 0.f, v2 = 0.f;
            const float* pk = a.pq + static_cast<size_t>(m) * nq + (a.H + kvh) * a.hd + i;
            const float* pv = a.pq + static_cast<size_t>(m) * nq + (a.H + a.Hkv + kvh) * a.hd + i;
            for (int s0 = 0; s0 < a.sp_q; s0 += 4) {
              float t[4][4];
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const bool in = s0 + u < a.sp_q;
                const size_t o = static_cast<size_t>(in ? s0 + u : 0) * kNT * nq;
                t[u][0] = in ? __ldcg(pk + o) : 0.f;
                t[u][1] = in ? __ldcg(pk + o + half) : 0.f;
                t[u][2] = in ? __ldcg(pv + o) : 0.f;
                t[u][3] = in ? __ldcg(pv + o + half) : 0.f;
              }
#pragma unroll
              for (int u = 0; u < 4; ++u) { k1 += t[u][0]; k2 += t[u][1]; v1 += t[u][2]; v2 += t[u][3]; }
            }
            const float2 c = cs[static_cast<size_t>(pos) * half + i];
            const int blk = a.kv.table[static_cast<size_t>(seq) * a.kv.bt_stride + (pos >> 4)];
            bf16* kd = poolw + (static_cast<size_t>(l) * a.kv.n_blocks + blk) * blk_stride + kvh * head_stride +
                       static_cast<size_t>(pos & 15) * a.hd;
            bf16* vd = kd + a.Hkv * head_stride;
            kd[i] = __float2bfloat16_rn(k1 * c.x - k2 * c.y);
            kd[i + half] = __float2bfloat16_rn(k2 * c.x + k1 * c.y);
            vd[i] = __float2bfloat16_rn(v1);
            vd[i + half] = __float2bfloat16_rn(v2);
          }
          __threadfence();
          asm volatile("bar.sync 1, 128;" ::: "memory");
          float m_run = -INFINITY, l_run = 0.f;
          const int NT2 = a.hd / 32;                 // n8 tiles of output dims per warp: 2 (hd 64) or 4
          float acc[4][4];
#pragma unroll
          for (int nt = 0; nt < 4; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;
          const float scale = rsqrtf(static_cast<float>(a.hd));
          const int srow = tid >> 2, squart = tid & 3;
          const bf16* layer_base = pool + static_cast<size_t>(l) * a.kv.n_blocks * blk_stride + kvh * head_stride;
          const int* table = a.kv.table + static_cast<size_t>(seq) * a.kv.bt_stride;
          for (int t0 = lo; t0 < hi; t0 += kTileP) {
            // K, V rows t0 .. t0+63 (zero past hi)
            const int cpr = a.hd / 8;
            for (int idx = tid; idx < kTileP * cpr; idx += 128) {
              const int t = idx / cpr, c = idx % cpr;
              const int p = t0 + t;
              uint4 kk = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
              if (p < hi) {
                const bf16* src = layer_base + static_cast<size_t>(table[p >> 4]) * blk_stride +
                                  static_cast<size_t>(p & 15) * a.hd + c * 8;
                kk = __ldcg(reinterpret_cast<const uint4*>(src));
                vv = __ldcg(reinterpret_cast<const uint4*>(src + a.Hkv * head_stride));
              }
              *reinterpret_cast<uint4*>(sK + t * KS + c * 8) = kk;
              *reinterpret_cast<uint4*>(sV + t * KS + c * 8) = vv;
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            // S = Q K^T: warp w4 owns positions 16 w4 .. 16 w4 + 15 (two n8 tiles)
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
              const int n0 = w4 * 16 + nt * 8;
              float c4[4] = {0.f, 0.f, 0.f, 0.f};
              for (int kk = 0; kk < a.hd / 16; ++kk) {
                const bf16* qa = sQ + g8 * KS + kk * 16 + 2 * t4;
                const bf16* kb = sK + (n0 + g8) * KS + kk * 16 + 2 * t4;
                const uint32_t a0 = *reinterpret_cast<const uint32_t*>(qa);
                const uint32_t a1 = *reinterpret_cast<const uint32_t*>(qa + 8 * KS);
                const uint32_t a2 = *reinterpret_cast<const uint32_t*>(qa + 8);
                const uint32_t a3 = *reinterpret_cast<const uint32_t*>(qa + 8 * KS + 8);
                const uint32_t b0 = *reinterpret_cast<const uint32_t*>(kb);
                const uint32_t b1 = *reinterpret_cast<const uint32_t*>(kb + 8);
                asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                    "{%0,%1,%2,%3};"
                    : "+f"(c4[0]), "+f"(c4[1]), "+f"(c4[2]), "+f"(c4[3])
                    : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
              }
              const int pc = t0 + n0 + 2 * t4;
              const int pa_ = sPos[g8], pb = sPos[g8 + 8];
              float2 s_a, s_b;
              s_a.x = (pc < hi && pc <= pa_) ? c4[0] * scale : -INFINITY;
              s_a.y = (pc + 1 < hi && pc + 1 <= pa_) ? c4[1] * scale : -INFINITY;
              s_b.x = (pc < hi && pc <= pb) ? c4[2] * scale : -INFINITY;
              s_b.y = (pc + 1 < hi && pc + 1 <= pb) ? c4[3] * scale : -INFINITY;
              *reinterpret_cast<float2*>(sS + g8 * SS + n0 + 2 * t4) = s_a;
              *reinterpret_cast<float2*>(sS + (g8 + 8) * SS + n0 + 2 * t4) = s_b;
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            // online softmax: 4 threads per query row (threads 0..63)
            if (tid < 64) {
              const float4* sr = reinterpret_cast<const float4*>(sS + srow * SS + squart * 16);
              float v[16];
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const float4 f = sr[i];
                v[4 * i] = f.x; v[4 * i + 1] = f.y; v[4 * i + 2] = f.z; v[4 * i + 3] = f.w;
              }
              float mx = v[0];
#pragma unroll
              for (int i = 1; i < 16; ++i) mx = fmaxf(mx, v[i]);
              mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
              mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
              const float m_new = fmaxf(m_run, mx);
              const float m_use = m_new == -INFINITY ? 0.f : m_new;
              const float corr = __expf(m_run - m_use);
              uint32_t pk[8];
              float sum = 0.f;
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const __nv_bfloat162 hb = __floats2bfloat162_rn(__expf(v[2 * i] - m_use), __expf(v[2 * i + 1] - m_use));
                sum += __low2float(hb) + __high2float(hb);
                pk[i] = *reinterpret_cast<const uint32_t*>(&hb);
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
            asm volatile("bar.sync 1, 128;" ::: "memory");
            // O = O * corr + P V: warp w4 owns output dims 8 NT2 w4 .. (NT2 n8 tiles)
            {
              const float ca = sCorr[g8], cb = sCorr[g8 + 8];
#pragma unroll
              for (int nt = 0; nt < 4; ++nt) {
                if (nt >= NT2) break;
                acc[nt][0] *= ca; acc[nt][1] *= ca; acc[nt][2] *= cb; acc[nt][3] *= cb;
              }
              for (int kk = 0; kk < kTileP / 16; ++kk) {
                const bf16* pa2 = sP + g8 * PS + kk * 16 + 2 * t4;
                const uint32_t a0 = *reinterpret_cast<const uint32_t*>(pa2);
                const uint32_t a1 = *reinterpret_cast<const uint32_t*>(pa2 + 8 * PS);
                const uint32_t a2 = *reinterpret_cast<const uint32_t*>(pa2 + 8);
                const uint32_t a3 = *reinterpret_cast<const uint32_t*>(pa2 + 8 * PS + 8);
#pragma unroll
                for (int nt = 0; nt < 4; ++nt) {
                  if (nt >= NT2) break;
                  const int d0 = (w4 * NT2 + nt) * 8;
                  const int row = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                  uint32_t b0, b1;
                  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];"
                               : "=r"(b0), "=r"(b1)
                               : "r"(smem_u32(sV + row * KS + d0))
                               : "memory");
                  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                      "{%0,%1,%2,%3};"
                      : "+f"(acc[nt][0]), "+f"(acc[nt][1]), "+f"(acc[nt][2]), "+f"(acc[nt][3])
                      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
                }
              }
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");   // the tile buffers are refilled next
          }
          // partial records Pa[split][m][h][hd + 2]: accumulator, running max, running sum
          if (tid < 64 && squart == 0) { sCorr[srow] = m_run; reinterpret_cast<float*>(sPos)[srow] = l_run; }
          asm volatile("bar.sync 1, 128;" ::: "memory");
#pragma unroll
          for (int half2 = 0; half2 < 2; ++half2) {
            const int qv = g8 + 8 * half2;
            if (qv >= nqv) continue;
            const int m = r0 + qv / G, hh = kvh * G + qv % G;
            float* rec = a.pa + ((static_cast<size_t>(split) * kNT + m) * a.H + hh) * (a.hd + 2);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
              if (nt >= NT2) break;
              const int dd = (w4 * NT2 + nt) * 8 + 2 * t4;
              rec[dd] = acc[nt][2 * half2];
              rec[dd + 1] = acc[nt][2 * half2 + 1];
            }
            if (w4 == 0 && t4 == 0) {
              rec[a.hd] = sCorr[qv];
              rec[a.hd + 1] = reinterpret_cast<float*>(sPos)[qv];
            }
          }
          asm volatile("bar.sync 1, 128;" ::: "memory");
        }
      }
      if (!(ok = grid_sync(a, bar_no++, abort_flag, ok_shared))) break;

      // ============================================================ O: merged attention -> Po
      {
        const Gemm g = gemm_of(a, 1);
        if (cta < g.tiles * g.sp) {
          const int sl = cta % g.sp, k0 = kb_lo(g, sl), k1 = kb_lo(g, sl + 1);
          const int c_lo = k0 * kBK, c_hi = k1 * kBK;
          const int h_lo = c_lo / a.hd, h_hi = (c_hi - 1) / a.hd + 1, nh = h_hi - h_lo;
          // split weights per (row, head): w_s = e^{m_s - max} / sum_s l_s e^{m_s - max}
          for (int e = tid; e < M * nh; e += 128) {
            const int m = e / nh, hh = h_lo + e % nh;
            const int ns = min(a.n_splits, a.row_pos[m] / a.chunk + 1);
            float ms[16], ls[16];                       // n_splits <= 16: every split's (max, sum) at once
#pragma unroll
            for (int s = 0; s < 16; ++s) {
              const float* rec = a.pa + ((static_cast<size_t>(s < ns ? s : 0) * kNT + m) * a.H + hh) * (a.hd + 2);
              ms[s] = s < ns ? __ldcg(rec + a.hd) : -INFINITY;
              ls[s] = s < ns ? __ldcg(rec + a.hd + 1) : 0.f;
            }
            float mx = -INFINITY;
#pragma unroll
            for (int s = 0; s < 16; ++s) mx = fmaxf(mx, ms[s]);
            float L = 0.f;
#pragma unroll
            for (int s = 0; s < 16; ++s) L += s < ns ? ls[s] * __expf(ms[s] - mx) : 0.f;
            wts[(m * 32 + (e % nh)) * 2] = mx;
            wts[(m * 32 + (e % nh)) * 2 + 1] = 1.f / L;
          }
          asm volatile("bar.sync 1, 128;" ::: "memory");
          for (int e = tid; e < kNT * (k1 - k0) * 8; e += 128) {
            const int m = e / ((k1 - k0) * 8), cc = e % ((k1 - k0) * 8);
            const int c = c_lo + cc * 8, kb = cc >> 3;
            uint4 o = make_uint4(0, 0, 0, 0);
            if (m < M) {
              const int hh = c / a.hd, dd = c % a.hd, hi2 = hh - h_lo;
              const int ns = min(a.n_splits, a.row_pos[m] / a.chunk + 1);
              const float mx = wts[(m * 32 + hi2) * 2], inv = wts[(m * 32 + hi2) * 2 + 1];
              float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
              for (int s0 = 0; s0 < ns; s0 += 4) {      // four splits' loads in flight at once
                float mw[4];
                float2 pr[4][4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                  const bool in = s0 + u < ns;
                  const float* rec = a.pa + ((static_cast<size_t>(in ? s0 + u : 0) * kNT + m) * a.H + hh) * (a.hd + 2);
                  mw[u] = in ? __ldcg(rec + a.hd) : -INFINITY;
#pragma unroll
                  for (int k2 = 0; k2 < 4; ++k2)
                    pr[u][k2] = in ? __ldcg(reinterpret_cast<const float2*>(rec + dd + 2 * k2)) : make_float2(0.f, 0.f);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                  const float w = __expf(mw[u] - mx) * inv;      // e^{-inf} = 0 past the last split
#pragma unroll
                  for (int k2 = 0; k2 < 4; ++k2) { v[2 * k2] += w * pr[u][k2].x; v[2 * k2 + 1] += w * pr[u][k2].y; }
                }
              }
              // the attention output is bf16 on the GEMM input side
              o = make_uint4(pack2(v[0], v[1]), pack2(v[2], v[3]), pack2(v[4], v[5]), pack2(v[6], v[7]));
            }
            *reinterpret_cast<uint4*>(breg + kb * kBBlock + sw_off(m, cc & 7)) = o;
          }
          b_ready();
          store_partial(a.po, a.d, cta / g.sp, sl);
          ++nb;
        }
      }
      if (!ok || !(ok = grid_sync(a, bar_no++, abort_flag, ok_shared))) break;

      // ============================================================ U: RMSNorm(x_l + sum Po) -> h
      {
        const Gemm g = gemm_of(a, 2);
        if (cta >= g.tiles) {                // no unit: only the owned columns of x'_l
          for (int m = 0; m < M; ++m) norm_build(m, xrow(a, 0, m), a.po, a.sp_o, 1, g_mlp, false, 0, 0);
        } else {
          for (int m = 0; m < kNT; ++m) {
            if (m >= M) {
              for (int cc = tid; cc < a.d / 8; cc += 128)
                *reinterpret_cast<uint4*>(breg + (cc >> 3) * kBBlock + sw_off(m, cc & 7)) = make_uint4(0, 0, 0, 0);
              continue;
            }
            norm_build(m, xrow(a, 0, m), a.po, a.sp_o, 1, g_mlp, true, 0, a.d / kBK);
          }
          for (int u = cta; u < g.tiles; u += a.n_cta) {
            if (u == cta) b_ready();
            else {                                   // the operand is the same: re-arm for the MMA thread
              asm volatile("bar.sync 1, 128;" ::: "memory");
              if (tid == 0) mbar_arrive(bready);
            }
            if (!wait_bar(tfull, nb & 1, abort_flag, a.err)) { ok = false; break; }
            tc_fence_after();
            float v[16];
            tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16), v);
            if (r >= 64)
#pragma unroll
              for (int m = 0; m < kNT; ++m) xch[(r - 64) * 17 + m] = v[m];
            tc_fence_before();
            asm volatile("bar.sync 1, 128;" ::: "memory");
            if (tid == 0) mbar_arrive(tempty);
            if (r < 64) {
              const int f = u * 64 + r;
#pragma unroll
              for (int m = 0; m < kNT; ++m) {
                if (m >= M) break;
                float up = xch[r * 17 + m];
                if (a.bias) up += a.bias[static_cast<size_t>(a.row_seq[m]) * a.ld_bias + static_cast<size_t>(l) * a.F + f];
                const float gate = v[m];
                a.h[static_cast<size_t>(m) * a.F + f] = __float2bfloat16_rn(up * (gate / (1.f + __expf(-gate))));
              }
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            ++nb;
          }
        }
      }
      if (!ok || !(ok = grid_sync(a, bar_no++, abort_flag, ok_shared))) break;

      // ============================================================ D: h -> Pd
      {
        const Gemm g = gemm_of(a, 3);
        if (cta < g.tiles * g.sp) {
          const int sl = cta % g.sp, k0 = kb_lo(g, sl), k1 = kb_lo(g, sl + 1);
          for (int e = tid; e < kNT * (k1 - k0) * 8; e += 128) {
            const int m = e / ((k1 - k0) * 8), cc = e % ((k1 - k0) * 8);
            uint4 o = make_uint4(0, 0, 0, 0);
            if (m < M) o = __ldcg(reinterpret_cast<const uint4*>(a.h + static_cast<size_t>(m) * a.F + k0 * kBK + cc * 8));
            *reinterpret_cast<uint4*>(breg + (cc >> 3) * kBBlock + sw_off(m, cc & 7)) = o;
          }
          b_ready();
          store_partial(a.pd, a.d, cta / g.sp, sl);
          ++nb;
        }
      }
    }
    // ============================================================ the residual stream after the last layer
    if (ok && grid_sync(a, bar_no++, abort_flag, ok_shared)) {
      for (int e = tid; e < M * (own_hi - own_lo) / 8; e += 128) {
        const int per = (own_hi - own_lo) / 8;
        const int m = e / per, c = own_lo + (e % per) * 8;
        float v[8], w[8];
        row_plus_slices(a, xrow(a, 1, m), a.pd, a.sp_d, m, c, c, false, v, w);
        float* xd = a.x_out + static_cast<size_t>(m) * a.d + c;
        *reinterpret_cast<float4*>(xd) = make_float4(v[0], v[1], v[2], v[3]);
        *reinterpret_cast<float4*>(xd + 4) = make_float4(v[4], v[5], v[6], v[7]);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 32);
}

// ------------------------------------------------------------------------------ host side
size_t align256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

}  // namespace

bool chain_plan(ChainPlan& p, int L, int d, int H, int Hkv, int hd, int F, int vocab, float eps, int max_splits) {
  p.L = L; p.d = d; p.H = H; p.Hkv = Hkv; p.hd = hd; p.F = F; p.vocab = vocab; p.eps = eps;
  p.max_splits = max_splits;
  if (hd != 64 && hd != 128) return false;
  // whole 128-row weight tiles in every segment (q, k, v, o, down); SwiGLU tiles of 64 features
  if (d % kW || d > kBRegion / (kNT * 2) || F % 64 || (H * hd) % kW || (Hkv * hd) % kW) return false;
  if (H % Hkv) return false;
  const int sms = sm_count_cached();
  p.n_cta = sms;
  auto split = [&](int tiles, int kb) {
    int sp = sms / tiles;
    if (sp > kb) sp = kb;
    if (sp > 32) sp = 32;
    return sp < 1 ? 1 : sp;
  };
  const int tq = (H + 2 * Hkv) * hd / kW, to = d / kW;
  p.sp_q = split(tq, d / kBK);
  p.sp_o = split(to, H * hd / kBK);
  p.sp_d = split(to, F / kBK);
  if (tq > sms || to > sms) return false;
  // one unit's K slice must fit the operand region
  if ((d / kBK + p.sp_q - 1) / p.sp_q > 32 || (H * hd / kBK + p.sp_o - 1) / p.sp_o > 32 ||
      (F / kBK + p.sp_d - 1) / p.sp_d > 32)
    return false;
  return true;
}

size_t chain_device_bytes(const ChainPlan& p) {
  size_t b = align256(sizeof(CUtensorMap) * kMaps * p.L) + align256(sizeof(void*) * 2 * p.L);
  const int nq = (p.H + 2 * p.Hkv) * p.hd;
  b += align256(4ull * 2 * kNT * p.d);
  b += align256(4ull * p.sp_q * kNT * nq);
  b += align256(4ull * p.sp_o * kNT * p.d);
  b += align256(4ull * p.sp_d * kNT * p.d);
  b += align256(4ull * p.max_splits * kNT * p.H * (p.hd + 2));
  b += align256(2ull * kNT * p.F);
  b += 256;
  return b;
}

cudaError_t chain_prepare(ChainPlan& p, const void* const* w, const void* embed, const KVCache& kv,
                          const float* rope_cs, void* block) {
  p.embed = embed;
  p.kv = kv;
  p.rope_cs = rope_cs;
  p.dev = block;
  std::vector<CUtensorMap> maps(static_cast<size_t>(kMaps) * p.L);
  std::vector<const void*> norms(2 * static_cast<size_t>(p.L));
  const int nqh = p.H * p.hd, nkv = p.Hkv * p.hd;
  for (int l = 0; l < p.L; ++l) {
    const void* const* lw = w + static_cast<size_t>(l) * SD2_LAYER_SLOTS;
    CUtensorMap* m = maps.data() + static_cast<size_t>(l) * kMaps;
    if (!encode_weight_map(m + 0, lw[SD2_W_Q], nqh, p.d, kW) || !encode_weight_map(m + 1, lw[SD2_W_K], nkv, p.d, kW) ||
        !encode_weight_map(m + 2, lw[SD2_W_V], nkv, p.d, kW) || !encode_weight_map(m + 3, lw[SD2_W_O], p.d, nqh, kW) ||
        !encode_weight_map(m + 4, lw[SD2_W_GATE], p.F, p.d, 64) || !encode_weight_map(m + 5, lw[SD2_W_UP], p.F, p.d, 64) ||
        !encode_weight_map(m + 6, lw[SD2_W_DOWN], p.d, p.F, kW))
      return cudaErrorInvalidValue;
    norms[2 * l] = lw[SD2_W_ATTN_NORM];
    norms[2 * l + 1] = lw[SD2_W_MLP_NORM];
  }
  unsigned char* b = static_cast<unsigned char*>(block);
  cudaError_t e = cudaMemcpy(b, maps.data(), sizeof(CUtensorMap) * maps.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return e;
  b += align256(sizeof(CUtensorMap) * kMaps * p.L);
  e = cudaMemcpy(b, norms.data(), sizeof(void*) * norms.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return e;
  b += align256(sizeof(void*) * 2 * p.L);
  const int nq = (p.H + 2 * p.Hkv) * p.hd;
  p.xbuf = reinterpret_cast<float*>(b); b += align256(4ull * 2 * kNT * p.d);
  p.pq = reinterpret_cast<float*>(b); b += align256(4ull * p.sp_q * kNT * nq);
  p.po = reinterpret_cast<float*>(b); b += align256(4ull * p.sp_o * kNT * p.d);
  p.pd = reinterpret_cast<float*>(b); b += align256(4ull * p.sp_d * kNT * p.d);
  p.pa = reinterpret_cast<float*>(b); b += align256(4ull * p.max_splits * kNT * p.H * (p.hd + 2));
  p.h = b; b += align256(2ull * kNT * p.F);
  p.sync = reinterpret_cast<unsigned*>(b);
  return cudaMemset(p.xbuf, 0, static_cast<size_t>(b - reinterpret_cast<unsigned char*>(p.xbuf)) + 256);
}

bool chain_supported(const ChainPlan& p, const ChainRun& r) {
  if (!p.dev || r.M < 1 || r.M > kNT || r.max_rows * (p.H / p.Hkv) > kQV) return false;
  if (r.n_splits < 1 || r.n_splits > p.max_splits || r.chunk % kTileP) return false;
  return true;
}

cudaError_t chain_forward(const ChainPlan& p, const ChainRun& r, cudaStream_t st) {
  if (!chain_supported(p, r)) return cudaErrorInvalidValue;
  ChainK a{};
  const unsigned char* b = static_cast<const unsigned char*>(p.dev);
  a.maps = reinterpret_cast<const CUtensorMap*>(b);
  a.norms = reinterpret_cast<const bf16* const*>(b + align256(sizeof(CUtensorMap) * kMaps * p.L));
  a.embed = static_cast<const bf16*>(p.embed);
  a.L = p.L; a.d = p.d; a.H = p.H; a.Hkv = p.Hkv; a.hd = p.hd; a.F = p.F; a.vocab = p.vocab; a.eps = p.eps;
  a.M = r.M;
  a.tok = r.tok; a.row_pos = r.row_pos; a.row_seq = r.row_seq; a.row_valid = r.row_valid;
  a.grp_row0 = r.grp_row0; a.grp_nrows = r.grp_nrows; a.grp_seq = r.grp_seq;
  a.n_groups = r.n_groups; a.n_splits = r.n_splits; a.chunk = r.chunk;
  a.kv = p.kv; a.rope_cs = p.rope_cs;
  a.bias = r.bias; a.ld_bias = r.ld_bias;
  a.x_out = r.x_out;
  a.xbuf = p.xbuf; a.pq = p.pq; a.po = p.po; a.pd = p.pd; a.pa = p.pa; a.h = static_cast<bf16*>(p.h);
  a.sync = p.sync; a.err = r.err;
  a.n_cta = p.n_cta; a.sp_q = p.sp_q; a.sp_o = p.sp_o; a.sp_d = p.sp_d;
  const int fixed = 1024 + kBRegion + 8 * (2 * 32 + 4) + (64 * 17 + 8 + 16 + 16 * 32 * 2) * 4 + 64;
  int S = (kSmem - fixed) / kAStage;
  if (S > 16) S = 16;
  if (S < 2) return cudaErrorInvalidValue;
  a.stages = S;
  const int smem = fixed + S * kAStage;
  static const cudaError_t configured =   // once per process (thread-safe initialisation)
      cudaFuncSetAttribute(chain_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (configured != cudaSuccess) return configured;
  cudaError_t e = cudaMemsetAsync(p.sync, 0, sizeof(unsigned), st);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.n_cta);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, chain_kernel, a);
}

}  // namespace sd2
