// Weight-streaming GEMM on the 5th-generation tensor cores: Y[m, n] = sum_k X[m, k] W[n, k] with
// the decoder's fused epilogues (store, residual add, steered SwiGLU of Eq. 2).
//
// The few token rows of a decode or verify step (M <= 256 per tile) cannot fill the M = 128
// side of tcgen05.mma, so the operands are swapped: each tile is 128 weight rows (the MMA's M)
// against NT token rows (the MMA's N, a multiple of 16), accumulating in TMEM. Weights and
// tokens are K-major bf16 tiles of 64 elements (128 bytes) per stage, loaded by TMA with the
// 128-byte swizzle that the UMMA shared-memory descriptors expect.
//
// Work split: the weight stream of a launch is U = tiles x (K/64) k-blocks; a persistent grid of
// G <= #SMs CTAs takes contiguous ranges of U/G k-blocks (stream-K), so every SM streams the same
// number of weight bytes whatever the matrix shape. A tile split across CTAs is finished by the
// last CTA to arrive on its counter, which sums the fp32 partials in k order (deterministic; no
// CTA ever waits on another).
//
// Warp roles (192 threads): warp 0 issues TMA loads into a ring of stages, warp 1 issues the
// MMAs (one thread) and owns the TMEM allocation, warps 2-5 read the two TMEM accumulators back
// (each warp its 32-lane quarter) and run the epilogue. Every wait is bounded by a clock budget;
// on expiry the kernel records ERR_TIMEOUT, drains what it issued and returns.
#include <cuda.h>

#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "kernels.h"

namespace sd2 {
namespace {

constexpr int kWRows = 128;          // weight rows per tile = the MMA's M
constexpr int kBK = 64;              // K per stage (128 bytes of bf16)
constexpr int kThreads = 192;
constexpr long long kWaitCycles = 4000000000ll;   // ~2 s at 2 GHz
constexpr long long kDrainCycles = 200000000ll;

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
  float* ws;
  int* counters;
  unsigned* err;
};

// ------------------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void named_bar_epi() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// UMMA shared-memory descriptor of a K-major tile with the 128-byte swizzle: rows of 128 bytes,
// 8-row groups 1024 bytes apart (stride byte offset), leading byte offset unused, version 1.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(1) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}
// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both K-major, M x N.
__device__ __forceinline__ uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

// Bounded wait on an mbarrier phase. Gives up when another role has aborted, or when the clock
// budget runs out (then records the timeout and raises the abort flag itself).
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int* abort_flag, unsigned* err) {
  if (mbar_try(bar, parity)) return true;
  const long long t0 = clock64();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try(bar, parity)) return true;
    if ((it & 31) == 0) {
      if (*abort_flag) return false;
      if (clock64() - t0 > kWaitCycles) {
        *abort_flag = 1;
        atomicOr(err, static_cast<unsigned>(ERR_TIMEOUT));
        return false;
      }
    }
  }
}
__device__ __forceinline__ bool wait_bar_budget(uint32_t bar, uint32_t parity, long long cycles) {
  const long long t0 = clock64();
  while (!mbar_try(bar, parity))
    if (clock64() - t0 > cycles) return false;
  return true;
}

struct Seg {
  int tile, kb, nkb;
};
__device__ __forceinline__ Seg segment(long long u, long long hi, int KB) {
  Seg s;
  s.tile = static_cast<int>(u / KB);
  s.kb = static_cast<int>(u % KB);
  s.nkb = static_cast<int>(min(static_cast<long long>(KB - s.kb), hi - u));
  return s;
}
__device__ __forceinline__ long long cta_lo(long long c, long long U, long long G) { return c * U / G; }
// The CTA whose range holds unit x (ranges are non-empty because G <= U).
__device__ __forceinline__ int cta_of(long long x, long long U, long long G) {
  long long c = x * G / U;
  while (c + 1 < G && cta_lo(c + 1, U, G) <= x) ++c;
  while (c > 0 && cta_lo(c, U, G) > x) --c;
  return static_cast<int>(c);
}

// Epilogue of 16 token columns j0..j0+15 of one weight row r of the tile.
__device__ __forceinline__ void finish_chunk(const TcArgs& a, int wt, int tt, int r, int j0, const float (&v)[16],
                                             float* xbuf) {
  const int m0 = tt * a.NT + j0;
  if (a.swiglu) {
    // rows 0..63: gate of feature f0 + r; rows 64..127: up of the same features
    constexpr int XS = 17;
    if (r >= 64)
#pragma unroll
      for (int j = 0; j < 16; ++j) xbuf[(r - 64) * XS + j] = v[j];
    named_bar_epi();
    if (r < 64) {
      const int f = wt * 64 + r;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int m = m0 + j;
        if (m < a.M) {
          float up = xbuf[r * XS + j];
          if (a.bias) up += a.bias[static_cast<size_t>(a.row_seq ? a.row_seq[m] : 0) * a.ld_bias + f];
          const float g = v[j];
          a.out_bf[static_cast<size_t>(m) * a.ldh + f] = __float2bfloat16_rn(up * (g / (1.f + __expf(-g))));
        }
      }
    }
    named_bar_epi();
    return;
  }
  const int n = wt * kWRows + r;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const int m = m0 + j;
    if (m < a.M) {
      float* o = a.out + static_cast<size_t>(m) * a.ldo + n;
      if (a.epi == EPI_ADD) *o += v[j];
      else *o = v[j];
    }
  }
}

__global__ void __launch_bounds__(kThreads, 2) gemm_tc_kernel(const __grid_constant__ TcArgs a) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = a.stages, NT = a.NT;
  const uint32_t a_bytes = kWRows * kBK * 2;
  const uint32_t b_bytes = static_cast<uint32_t>(NT) * kBK * 2;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(S) * stage_bytes);
  // bars: full[S], empty[S], tfull[2], tempty[2], drain
  float* xbuf = reinterpret_cast<float*>(bars + 2 * S + 6);
  volatile int* flags = reinterpret_cast<volatile int*>(xbuf + 64 * 17);
  // flags: [0] abort, [1] TMEM base, [2] last-arrival decision, [3] stages consumed, [4] go
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, tfull0 = empty0 + 8 * S, tempty0 = tfull0 + 16,
                 drain = tempty0 + 16;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t ncols = 32;
  while (ncols < static_cast<uint32_t>(2 * NT)) ncols <<= 1;

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
    flags[0] = 0; flags[2] = 0; flags[3] = 0; flags[4] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<int*>(flags) + 1), ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = static_cast<uint32_t>(flags[1]);

  const long long G = gridDim.x, U = a.units, c = blockIdx.x;
  const long long lo = cta_lo(c, U, G), hi = cta_lo(c + 1, U, G);
  volatile int* abort_flag = flags;

  pdl_trigger();                             // the next kernel may start its own prologue
  if (warp == 0) {
    if (lane == 0) {
      // Stage use j loads k-block (lo + j) of this CTA's range: the weight half first, then the
      // token half. Weights never depend on earlier kernels, so the first stages' weight tiles
      // are requested before waiting for the predecessor grid. Cursors advance one k-block at a
      // time (no divisions in the issue loop: this one thread feeds the whole SM).
      const uint32_t n_units = static_cast<uint32_t>(hi - lo);
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
        if (++c.kb == a.KB) { c.kb = 0; ++c.tile; locate(c); }
      };
      Cursor ca, cb;
      ca.tile = static_cast<int>(lo / a.KB);
      ca.kb = static_cast<int>(lo % a.KB);
      locate(ca);
      cb = ca;
      auto load_a = [&](uint32_t j, const Cursor& c) {
        const uint32_t s = j % S;
        const uint32_t dst = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
        if (a.swiglu) {
          tma_load_2d(dst, &a.mapA[0], c.kb * kBK, c.wt * 64, full0 + 8 * s);
          tma_load_2d(dst + a_bytes / 2, &a.mapA[1], c.kb * kBK, c.wt * 64, full0 + 8 * s);
        } else {
          tma_load_2d(dst, &a.mapA[c.seg], c.kb * kBK, c.row0, full0 + 8 * s);
        }
      };
      auto load_b = [&](uint32_t j, const Cursor& c) {
        const uint32_t s = j % S;
        const uint32_t dst = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
        tma_load_2d(dst + a_bytes, &a.mapB, c.kb * kBK, c.tt * NT, full0 + 8 * s);
      };
      const uint32_t pre = n_units < static_cast<uint32_t>(S) ? n_units : static_cast<uint32_t>(S);
      for (uint32_t j = 0; j < pre; ++j, advance(ca)) {   // first use of each stage: no wait
        mbar_expect_tx(full0 + 8 * j, stage_bytes);
        load_a(j, ca);
      }
      pdl_wait();
      for (uint32_t j = 0; j < pre; ++j, advance(cb)) load_b(j, cb);
      uint32_t j = pre;
      bool ok = true;
      for (; j < n_units; ++j, advance(ca)) {
        const uint32_t s = j % S;
        if (!wait_bar(empty0 + 8 * s, ((j / S) & 1) ^ 1, abort_flag, a.err)) { ok = false; break; }
        mbar_expect_tx(full0 + 8 * s, stage_bytes);
        load_a(j, ca);
        load_b(j, ca);
      }
      if (!ok) {  // let the loads already issued land before the CTA exits
        const uint32_t done = static_cast<uint32_t>(flags[3]);
        for (uint32_t jj = done; jj < j; ++jj) wait_bar_budget(full0 + 8 * (jj % S), (jj / S) & 1, kDrainCycles);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kWRows, NT);
      uint32_t j = 0, segi = 0;
      bool ok = true;
      for (long long u = lo; u < hi && ok; ++segi) {
        const Seg sg = segment(u, hi, a.KB);
        const uint32_t acc = segi & 1;
        if (!wait_bar(tempty0 + 8 * acc, ((segi >> 1) & 1) ^ 1, abort_flag, a.err)) break;
        tc_fence_after();
        const uint32_t d = tmem + acc * NT;
        for (int i = 0; i < sg.nkb; ++i, ++j) {
          const uint32_t s = j % S;
          if (!wait_bar(full0 + 8 * s, (j / S) & 1, abort_flag, a.err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t abase = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
          const uint64_t ad = sw128_desc(abase), bd = sw128_desc(abase + a_bytes);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            mma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
          mma_commit(empty0 + 8 * s);
          flags[3] = static_cast<int>(j + 1);
        }
        if (!ok) break;
        mma_commit(tfull0 + 8 * acc);
        u += sg.nkb;
      }
      mma_commit(drain);                      // all MMAs issued by this thread have completed
      wait_bar_budget(drain, 0, kDrainCycles);
    }
    __syncwarp();
  } else {
    const int q = warp & 3;                   // TMEM lane quarter of this warp
    const int r = q * 32 + lane;              // weight row within the tile
    const bool leader = (warp == 2 && lane == 0);
    pdl_wait();                              // outputs, residuals and biases come from earlier kernels
    uint32_t segi = 0;
    for (long long u = lo; u < hi; ++segi) {
      const Seg sg = segment(u, hi, a.KB);
      const uint32_t acc = segi & 1;
      if (leader) flags[4] = wait_bar(tfull0 + 8 * acc, (segi >> 1) & 1, abort_flag, a.err) ? 1 : 0;
      named_bar_epi();
      const bool go = flags[4] != 0;
      tc_fence_after();
      if (!go) break;
      const int wt = sg.tile % a.n_wtiles, tt = sg.tile / a.n_wtiles;
      const uint32_t tbase = tmem + (static_cast<uint32_t>(q * 32) << 16) + acc * NT;
      const bool full_tile = (sg.kb == 0 && sg.nkb == a.KB);
      const int nchunk = NT / 16;
      const int rows_left = a.M - tt * NT;    // token columns of this tile that exist
      if (full_tile) {
        for (int ch = 0; ch < nchunk; ++ch) {
          if (ch * 16 >= rows_left) break;
          float v[16];
          tmem_ld16(tbase + ch * 16, v);
          finish_chunk(a, wt, tt, r, ch * 16, v, xbuf);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
      } else {
        // partial of a split tile: store it, then the last CTA to arrive sums them in k order
        const int slot = (u == lo) ? 0 : 1;
        float* wsrow = a.ws + ((static_cast<size_t>(c) * 2 + slot) * kWRows + r) * NT;
        for (int ch = 0; ch < nchunk; ++ch) {
          float v[16];
          tmem_ld16(tbase + ch * 16, v);
#pragma unroll
          for (int j = 0; j < 16; j += 4)
            *reinterpret_cast<float4*>(wsrow + ch * 16 + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
        const long long t_lo = static_cast<long long>(sg.tile) * a.KB, t_hi = t_lo + a.KB;
        const int c1 = cta_of(t_lo, U, G), c2 = cta_of(t_hi - 1, U, G);
        named_bar_epi();                       // every partial row of this CTA is written
        if (leader) {
          __threadfence();                     // release them (cumulative over the barrier)
          const int old = atomicAdd(&a.counters[sg.tile], 1);
          const bool last = (old == c2 - c1);
          if (last) a.counters[sg.tile] = 0;
          __threadfence();                     // acquire the other CTAs' partials
          flags[2] = last ? 1 : 0;
        }
        named_bar_epi();
        if (flags[2]) {
          for (int ch = 0; ch < nchunk; ++ch) {
            if (ch * 16 >= rows_left) break;
            float v[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = 0.f;
#pragma unroll 8
            for (int cc = c1; cc <= c2; ++cc) {
              const int sl = (cta_lo(cc, U, G) / a.KB == sg.tile) ? 0 : 1;
              const float* src = a.ws + ((static_cast<size_t>(cc) * 2 + sl) * kWRows + r) * NT + ch * 16;
#pragma unroll
              for (int j = 0; j < 16; j += 4) {
                const float4 t = __ldcg(reinterpret_cast<const float4*>(src + j));
                v[j] += t.x; v[j + 1] += t.y; v[j + 2] += t.z; v[j + 3] += t.w;
              }
            }
            finish_chunk(a, wt, tt, r, ch * 16, v, xbuf);
          }
        }
        named_bar_epi();
      }
      u += sg.nkb;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, ncols);
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

}  // namespace

int gemm_tc_token_tile(int M) {
  int nt = ((M + 15) / 16) * 16;
  return nt > 256 ? 256 : (nt < 16 ? 16 : nt);
}

size_t gemm_tc_workspace_floats(int max_M) {
  return static_cast<size_t>(512) * 2 * kWRows * gemm_tc_token_tile(max_M);
}

bool gemm_tc_supported(const GemmArgs& g) {
  if (g.K % kBK != 0 || g.K < kBK || g.M < 1 || g.ldx % 8 != 0) return false;
  if (reinterpret_cast<uintptr_t>(g.x) & 15) return false;
  if (g.epi == EPI_SWIGLU) return g.nseg == 2 && g.seg[0].rows == g.seg[1].rows && g.seg[0].rows % 64 == 0;
  for (int s = 0; s < g.nseg; ++s)
    if (g.seg[s].rows % kWRows != 0) return false;
  return true;
}

cudaError_t gemm_tc(const GemmArgs& g, float* ws, int* counters, size_t counters_len, unsigned* err,
                    cudaStream_t st) {
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
  const long long tiles = static_cast<long long>(a.n_wtiles) * a.n_ttiles;
  if (static_cast<size_t>(tiles) > counters_len) return cudaErrorInvalidValue;
  a.units = tiles * a.KB;
  a.epi = g.epi; a.out = g.out; a.ldo = g.ldo; a.out_bf = static_cast<bf16*>(g.out_bf); a.ldh = g.ldh;
  a.bias = g.bias; a.ld_bias = g.ld_bias; a.row_seq = g.row_seq;
  a.ws = ws; a.counters = counters; a.err = err;
  const int stage_bytes = (kWRows + a.NT) * kBK * 2;
  const int fixed = 1024 + 64 * 17 * 4 + 64 + 8 * (2 * 16 + 6);
  // Up to NT = 128 the ring fits in half an SM's shared memory (and the two accumulators in half
  // of TMEM), so the next GEMM's CTA can start on the same SM while this one drains.
  int S = (kSmemShared - fixed) / stage_bytes;
  if (a.NT > 128 || S < 3) S = (kSmemBudget - fixed) / stage_bytes;
  if (S > 8) S = 8;
  if (S < 2) return cudaErrorInvalidValue;
  a.stages = S;
  const int smem = fixed + S * stage_bytes;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  // At least kMinUnits k-blocks (kMinUnits x 16 KB of weights) per CTA: fewer CTAs share a
  // tile, so the last one to arrive sums fewer partials.
  constexpr long long kMinUnits = 8;
  long long G = sm_count();
  const long long g_cap = (a.units + kMinUnits - 1) / kMinUnits;
  if (G > g_cap) G = g_cap;
  if (G > a.units) G = a.units;
  if (G > 512) G = 512;
  return launch_pdl(gemm_tc_kernel, dim3(static_cast<unsigned>(G)), dim3(kThreads), static_cast<size_t>(smem), st, a);
}

}  // namespace sd2
