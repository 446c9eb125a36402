// Device helpers shared by the SD^2 kernels: bf16 conversion, warp/block reductions,
// Philox4x32-10, the exp/log used by every sampling decision, and order-preserving keys for
// deterministic atomic arg-max.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace sd2 {

typedef __nv_bfloat16 bf16;

// ------------------------------------------------------------------------------------------
// Loads
// ------------------------------------------------------------------------------------------

// 16-byte load that bypasses L1 allocation: weights are streamed once per launch.
__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float bf2f(bf16 v) { return __bfloat162float(v); }

// ------------------------------------------------------------------------------------------
// Reductions
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    unsigned long long t = __shfl_xor_sync(0xffffffffu, v, o);
    v = t > v ? t : v;
  }
  return v;
}
__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide sum of one float per thread (blockDim.x multiple of 32, <= 1024).
__device__ __forceinline__ float block_sum(float v, float* red32) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
  __syncthreads();
  if (l == 0) red32[w] = v;
  __syncthreads();
  v = (l < nw) ? red32[l] : 0.f;
  return warp_sum(v);
}

// ------------------------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): 10 rounds of multiply-high/low mixing of
// a 4x32-bit counter under a 2x32-bit key advanced by Weyl constants between rounds.
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// Purposes of the random draws (second counter word, bits 16 and up).
enum { RNG_DRAFT = 0, RNG_ACCEPT = 1, RNG_RESAMPLE = 2 };

// u = (2*(x >> 9) + 1) * 2^-24: an odd multiple of 2^-24 in (0,1), exact in fp32.
__device__ __forceinline__ float bits_to_u01(uint32_t x) {
  return __fmul_rn(__uint2float_rn(((x >> 9) << 1) | 1u), 0x1p-24f);
}

// ------------------------------------------------------------------------------------------
// exp and log for the sampling decisions, as fixed sequences of correctly rounded fp32
// operations (no contraction: every step is an explicit _rn intrinsic), so that a host
// implementation of the same methods reaches the same bits.
//   exp: Cody & Waite reduction n = rint(t/ln2), r = t - n*ln2_hi - n*ln2_lo, degree-7 Taylor
//        polynomial of e^r in Horner form (coefficients 1/j! rounded to fp32), times 2^n;
//        t < -80 gives 0.
//   log: x = 2^e m, m in [sqrt(1/2), sqrt(2)); ln m = 2 atanh(s), s = (m-1)/(m+1), by the odd
//        series 2(s + s^3/3 + ... + s^11/11) (Abramowitz & Stegun 4.1.27); ln x = e*ln2_hi +
//        (e*ln2_lo + ln m).
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ float exp_cw(float t) {
  if (t < -80.0f) return 0.0f;
  // n = rint(t / ln2) by adding and subtracting 1.5 * 2^23 (exact round-half-even for |t / ln2| <
  // 2^22; here t <= 0 and t / ln2 >= -116); the integer n sits in the low mantissa bits of the sum.
  const float nm = __fadd_rn(__fmul_rn(t, 0x1.715476p+0f), 0x1.8p+23f);
  const float n = __fsub_rn(nm, 0x1.8p+23f);
  const int ni = __float_as_int(nm) - 0x4B400000;
  float r = __fsub_rn(t, __fmul_rn(n, 0x1.62e400p-1f));
  r = __fsub_rn(r, __fmul_rn(n, 0x1.7f7d1cp-20f));
  float p = 0x1.a01a02p-13f;
  p = __fadd_rn(__fmul_rn(p, r), 0x1.6c16c2p-10f);
  p = __fadd_rn(__fmul_rn(p, r), 0x1.111112p-7f);
  p = __fadd_rn(__fmul_rn(p, r), 0x1.555556p-5f);
  p = __fadd_rn(__fmul_rn(p, r), 0x1.555556p-3f);
  p = __fadd_rn(__fmul_rn(p, r), 0x1p-1f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  // p in [0.7, 1.5] and n >= -116: adding n to the exponent field is the exact scaling by 2^n.
  return __int_as_float(__float_as_int(p) + ni * (1 << 23));
}

__device__ __forceinline__ float log_at(float x) {
  const uint32_t b = __float_as_uint(x);
  int e = static_cast<int>(b >> 23) - 127;
  float m = __uint_as_float((b & 0x7FFFFFu) | 0x3F800000u);
  if (m > 0x1.6a09e6p+0f) { m = __fmul_rn(m, 0.5f); e += 1; }
  const float s = __fdiv_rn(__fsub_rn(m, 1.0f), __fadd_rn(m, 1.0f));
  const float s2 = __fmul_rn(s, s);
  float q = 0x1.745d18p-4f;
  q = __fadd_rn(__fmul_rn(q, s2), 0x1.c71c72p-4f);
  q = __fadd_rn(__fmul_rn(q, s2), 0x1.24924ap-3f);
  q = __fadd_rn(__fmul_rn(q, s2), 0x1.99999ap-3f);
  q = __fadd_rn(__fmul_rn(q, s2), 0x1.555556p-2f);
  const float two_s = __fmul_rn(s, 2.0f);
  const float ln_m = __fadd_rn(two_s, __fmul_rn(two_s, __fmul_rn(s2, q)));
  const float ef = static_cast<float>(e);
  return __fadd_rn(__fmul_rn(ef, 0x1.62e400p-1f), __fadd_rn(__fmul_rn(ef, 0x1.7f7d1cp-20f), ln_m));
}

// e in [0, 1] to the fixed point floor(e * 2^45) of the exact softmax normaliser (the sum over the
// vocabulary of floor(e_v 2^45) is an integer, so its value does not depend on the summation
// order), as two exact 32-bit parts: floor(e 2^45) = hi 2^23 + lo with hi = floor(e 2^22) (<= 2^22)
// and lo = floor(e 2^45 - hi 2^23) (< 2^23). Every fp32 operation here is exact: the floors are
// round-toward-zero additions of 2^23 whose integer is read from the sum's bits, and
// e 2^45 - hi 2^23 is a multiple of the ulp of e 2^45 below 2^23. Sums of up to 2^9 parts fit in
// 32 bits. (A float-to-64-bit conversion would run on the FP64 pipe.)
__device__ __forceinline__ void fixed45_parts(float e, uint32_t& hi, uint32_t& lo) {
  const float h = __fadd_rz(__fmul_rn(e, 0x1p22f), 0x1p23f);
  hi = __float_as_uint(h) - 0x4B000000u;
  const float r = __fmaf_rn(-__fsub_rn(h, 0x1p23f), 0x1p23f, __fmul_rn(e, 0x1p45f));
  lo = __float_as_uint(__fadd_rz(r, 0x1p23f)) - 0x4B000000u;
}

// ------------------------------------------------------------------------------------------
// Order-preserving 32-bit code of a float (for atomicMax); -0 is folded onto +0 first so that
// equal values compare equal. Packed with the index so the maximum takes the lowest index.
// ------------------------------------------------------------------------------------------

__device__ __forceinline__ uint32_t ord_f32(float f) {
  const uint32_t b = __float_as_uint(__fadd_rn(f, 0.0f));
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float unord_f32(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}
__device__ __forceinline__ unsigned long long pack_key(float key, uint32_t idx) {
  return (static_cast<unsigned long long>(ord_f32(key)) << 32) | (0xFFFFFFFFu - idx);
}
__device__ __forceinline__ uint32_t packed_index(unsigned long long p) {
  return 0xFFFFFFFFu - static_cast<uint32_t>(p & 0xFFFFFFFFull);
}
__device__ __forceinline__ float packed_key(unsigned long long p) {
  return unord_f32(static_cast<uint32_t>(p >> 32));
}

// ------------------------------------------------------------------------------------------
// Programmatic dependent launch: every kernel of the hot path is launched so that it may start
// while its predecessor finishes. pdl_trigger lets the successor be scheduled; pdl_wait blocks
// until the predecessor grid has completed and its writes are visible. A kernel touches no
// global memory written by earlier kernels, and writes none, before pdl_wait.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ------------------------------------------------------------------------------------------
// Thread-block clusters: rank, full barrier (release/acquire), and loads from the shared memory
// of another CTA of the cluster (distributed shared memory).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// The two halves of a cluster barrier: every thread of the cluster arrives once (relaxed: after
// the mbarrier initialisation fence) and waits once, later.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
__device__ __forceinline__ uint32_t dsmem_addr(uint32_t saddr, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(saddr), "r"(rank));
  return remote;
}
// fp32 at shared-memory address `saddr` of CTA `rank` of this cluster
__device__ __forceinline__ float ld_dsmem(uint32_t saddr, uint32_t rank) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(dsmem_addr(saddr, rank)) : "memory");
  return v;
}
// four fp32 (16-byte aligned) at `saddr` of CTA `rank`
__device__ __forceinline__ float4 ld_dsmem_v4(uint32_t saddr, uint32_t rank) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(dsmem_addr(saddr, rank))
               : "memory");
  return v;
}

// four fp32 stored to `saddr` (16-byte aligned) of CTA `rank`
__device__ __forceinline__ void st_dsmem_v4(uint32_t saddr, uint32_t rank, float x, float y, float z, float w) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(dsmem_addr(saddr, rank)), "f"(x), "f"(y),
               "f"(z), "f"(w)
               : "memory");
}

// four fp32 stored asynchronously to `raddr` (a shared::cluster address, 16-byte aligned); the
// store's 16 bytes complete a transaction on the mbarrier at `rbar` (shared::cluster, same CTA)
__device__ __forceinline__ void st_async_v4(uint32_t raddr, uint32_t rbar, float x, float y, float z, float w) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(raddr),
               "f"(x), "f"(y), "f"(z), "f"(w), "r"(rbar)
               : "memory");
}

// Device error word bits (latched; read and cleared by the host).
enum { ERR_NONFINITE = 1, ERR_TIMEOUT = 2, ERR_RANGE = 4 };

}  // namespace sd2
