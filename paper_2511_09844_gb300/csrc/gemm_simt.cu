// Weight-streaming GEMM on the CUDA cores: Y = X W^T for few token rows (M small), with the
// decoder's epilogues fused (store, residual add, steered SwiGLU of Eq. 2).
//
// Each warp owns two weight rows (for the SwiGLU epilogue: row f of W_gate and row f of W_up)
// and streams them once per pass of up to 8 token rows with 16-byte non-allocating loads; the
// token rows come through L1. Partial dot products are reduced across the warp and one lane
// per token row runs the epilogue.
#include "common.cuh"
#include "kernels.h"

namespace sd2 {
namespace {

constexpr int kThreads = 256;
constexpr int kRowsPerPass = 8;

__device__ __forceinline__ void unpack8(const uint4 v, float f[8]) {
  f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
  f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
}

__device__ __forceinline__ const bf16* seg_row(const GemmArgs& a, int n) {
  int base = 0;
#pragma unroll
  for (int s = 0; s < 3; ++s) {
    if (s < a.nseg && n < base + a.seg[s].rows)
      return static_cast<const bf16*>(a.seg[s].w) + static_cast<size_t>(n - base) * a.K;
    base += a.seg[s].rows;
  }
  return nullptr;
}

template <int EPI>
__global__ void __launch_bounds__(kThreads) gemm_simt_kernel(const GemmArgs a, int n_units, int n_total) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int n_warps = (gridDim.x * kThreads) >> 5;
  const bf16* x = static_cast<const bf16*>(a.x);

  for (int u = warp; u < n_units; u += n_warps) {
    const bf16 *w0, *w1;
    int n0, n1;
    if (EPI == EPI_SWIGLU) {
      n0 = n1 = u;
      w0 = static_cast<const bf16*>(a.seg[0].w) + static_cast<size_t>(u) * a.K;
      w1 = static_cast<const bf16*>(a.seg[1].w) + static_cast<size_t>(u) * a.K;
    } else {
      n0 = 2 * u;
      n1 = (2 * u + 1 < n_total) ? 2 * u + 1 : -1;
      w0 = seg_row(a, n0);
      w1 = n1 >= 0 ? seg_row(a, n1) : nullptr;
    }
    for (int m0 = 0; m0 < a.M; m0 += kRowsPerPass) {
      float acc0[kRowsPerPass], acc1[kRowsPerPass];
#pragma unroll
      for (int m = 0; m < kRowsPerPass; ++m) acc0[m] = acc1[m] = 0.f;
#pragma unroll 2
      for (int k = lane * 8; k < a.K; k += 256) {
        float fa[8], fb[8];
        unpack8(ld_stream(w0 + k), fa);
        if (w1) unpack8(ld_stream(w1 + k), fb);
        else {
#pragma unroll
          for (int j = 0; j < 8; ++j) fb[j] = 0.f;
        }
#pragma unroll
        for (int m = 0; m < kRowsPerPass; ++m) {
          if (m0 + m < a.M) {
            float xf[8];
            unpack8(__ldg(reinterpret_cast<const uint4*>(x + static_cast<size_t>(m0 + m) * a.ldx + k)), xf);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              acc0[m] = fmaf(fa[j], xf[j], acc0[m]);
              acc1[m] = fmaf(fb[j], xf[j], acc1[m]);
            }
          }
        }
      }
      float v0 = 0.f, v1 = 0.f;
#pragma unroll
      for (int m = 0; m < kRowsPerPass; ++m) {
        const float s0 = warp_sum(acc0[m]);
        const float s1 = warp_sum(acc1[m]);
        if (lane == m) { v0 = s0; v1 = s1; }
      }
      const int m = m0 + lane;
      if (lane < kRowsPerPass && m < a.M) {
        if (EPI == EPI_STORE) {
          a.out[static_cast<size_t>(m) * a.ldo + n0] = v0;
          if (n1 >= 0) a.out[static_cast<size_t>(m) * a.ldo + n1] = v1;
        } else if (EPI == EPI_ADD) {
          if (a.bias) {   // a bias of the row's sequence added with the output (after-MLP steering)
            const float* bs = a.bias + static_cast<size_t>(a.row_seq ? a.row_seq[m] : 0) * a.ld_bias;
            v0 += bs[n0];
            if (n1 >= 0) v1 += bs[n1];
          }
          a.out[static_cast<size_t>(m) * a.ldo + n0] += v0;
          if (n1 >= 0) a.out[static_cast<size_t>(m) * a.ldo + n1] += v1;
        } else if (EPI == EPI_SILU) {
          bf16* hb = static_cast<bf16*>(a.out_bf) + static_cast<size_t>(m) * a.ldh;
          const float* bs = a.bias ? a.bias + static_cast<size_t>(a.row_seq ? a.row_seq[m] : 0) * a.ld_bias : nullptr;
          const float y0 = v0 + (bs ? bs[n0] : 0.f);
          hb[n0] = __float2bfloat16_rn(y0 / (1.f + __expf(-y0)));
          if (n1 >= 0) {
            const float y1 = v1 + (bs ? bs[n1] : 0.f);
            hb[n1] = __float2bfloat16_rn(y1 / (1.f + __expf(-y1)));
          }
        } else {
          float up = v1;
          if (a.bias) {
            const int s = a.row_seq ? a.row_seq[m] : 0;
            up += a.bias[static_cast<size_t>(s) * a.ld_bias + u];
          }
          const float h = up * (v0 / (1.f + __expf(-v0)));
          static_cast<bf16*>(a.out_bf)[static_cast<size_t>(m) * a.ldh + u] = __float2bfloat16_rn(h);
        }
      }
    }
  }
}

}  // namespace

// Token rows above which the tensor-core QKV projection stores plain q/k/v and a separate kernel
// rotates and appends them: the fused epilogue fetches each output's rotary factors and cache
// block from global memory, and with this many token columns per tile those dependent loads
// (several rounds per owner thread) cost more than one extra elementwise kernel.
constexpr int kQkvFusedMaxRows = 64;

cudaError_t gemm(const GemmArgs& a, cudaStream_t st) {
  if (a.attn_q) return a.impl != 1 && a.err && gemm_attn_supported(a) ? gemm_tc(a, a.err, st) : cudaErrorNotSupported;
  if (a.impl != 1 && a.err && a.epi == EPI_QKV && a.M > kQkvFusedMaxRows) {
    GemmArgs s = a;
    s.epi = EPI_STORE;
    if (gemm_tc_supported(s)) {
      cudaError_t e = gemm_tc(s, a.err, st);
      if (e != cudaSuccess) return e;
      KVCache kv;
      kv.pool = a.kv_pool; kv.table = a.kv_table; kv.bt_stride = a.kv_bt_stride; kv.n_blocks = a.kv_n_blocks;
      kv.Hkv = a.n_kv_heads; kv.hd = a.head_dim;
      return rope_append(a.out, a.rope_cs, a.M, a.n_heads, a.n_kv_heads, a.head_dim, a.row_seq, a.row_pos,
                         a.row_valid, kv, a.layer, a.q_out, st);
    }
  }
  if (a.impl != 1 && a.err && gemm_tc_supported(a)) return gemm_tc(a, a.err, st);
  if (a.norm_out || a.norm_ssq_in) return cudaErrorNotSupported;  // the fused RMSNorm is tensor-core only
  if (a.epi != EPI_QKV) return gemm_simt(a, st);
  // CUDA-core path of the QKV epilogue: projections to `out`, then the rotary/append kernel
  GemmArgs s = a;
  s.epi = EPI_STORE;
  cudaError_t e = gemm_simt(s, st);
  if (e != cudaSuccess) return e;
  KVCache kv;
  kv.pool = a.kv_pool; kv.table = a.kv_table; kv.bt_stride = a.kv_bt_stride; kv.n_blocks = a.kv_n_blocks;
  kv.Hkv = a.n_kv_heads; kv.hd = a.head_dim;
  return rope_append(a.out, a.rope_cs, a.M, a.n_heads, a.n_kv_heads, a.head_dim, a.row_seq, a.row_pos, a.row_valid, kv,
                     a.layer, a.q_out, st);
}

cudaError_t gemm_simt(const GemmArgs& a, cudaStream_t st) {
  int n_total = 0;
  for (int s = 0; s < a.nseg; ++s) n_total += a.seg[s].rows;
  const int n_units = (a.epi == EPI_SWIGLU) ? a.seg[0].rows : (n_total + 1) / 2;
  if (n_units <= 0 || a.M <= 0) return cudaSuccess;
  int blocks = (n_units * 32 + kThreads - 1) / kThreads;
  const int cap = 152 * 8;
  if (blocks > cap) blocks = cap;
  switch (a.epi) {
    case EPI_QKV:
    case EPI_STORE: { const cudaError_t e_ = launch_pdl(gemm_simt_kernel<EPI_STORE>, dim3(blocks), dim3(kThreads), 0, st, a, n_units, n_total); if (e_ != cudaSuccess) return e_; } break;
    case EPI_ADD: { const cudaError_t e_ = launch_pdl(gemm_simt_kernel<EPI_ADD>, dim3(blocks), dim3(kThreads), 0, st, a, n_units, n_total); if (e_ != cudaSuccess) return e_; } break;
    case EPI_SILU: { const cudaError_t e_ = launch_pdl(gemm_simt_kernel<EPI_SILU>, dim3(blocks), dim3(kThreads), 0, st, a, n_units, n_total); if (e_ != cudaSuccess) return e_; } break;
    default: { const cudaError_t e_ = launch_pdl(gemm_simt_kernel<EPI_SWIGLU>, dim3(blocks), dim3(kThreads), 0, st, a, n_units, n_total); if (e_ != cudaSuccess) return e_; } break;
  }
  return cudaGetLastError();
}

}  // namespace sd2
