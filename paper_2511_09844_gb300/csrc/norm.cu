// Row-wise decoder kernels: embedding + RMSNorm, RMSNorm with hidden-state taps, rotary
// embedding with the paged KV append, the steering vector's layer norm (App. A.2), the steered
// SwiGLU of Eq. 2 on precomputed projections, and the f32 -> bf16 row gather of the taps.
#include "common.cuh"
#include "kernels.h"

namespace sd2 {
namespace {

constexpr int kNormThreads = 256;

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ float row_inv_rms(const float* xr, int d, float eps, float* red) {
  float ss = 0.f;
  for (int j = threadIdx.x * 4; j < d; j += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = block_sum(ss, red);
  return rsqrtf(ss / static_cast<float>(d) + eps);
}

__device__ __forceinline__ void write_normed(const float* xr, const bf16* gamma, float inv, int d, bf16* out) {
  for (int j = threadIdx.x * 4; j < d; j += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    const __nv_bfloat162 g01 = *reinterpret_cast<const __nv_bfloat162*>(gamma + j);
    const __nv_bfloat162 g23 = *reinterpret_cast<const __nv_bfloat162*>(gamma + j + 2);
    __nv_bfloat162 o01 = __floats2bfloat162_rn(v.x * inv * __low2float(g01), v.y * inv * __high2float(g01));
    __nv_bfloat162 o23 = __floats2bfloat162_rn(v.z * inv * __low2float(g23), v.w * inv * __high2float(g23));
    *reinterpret_cast<__nv_bfloat162*>(out + j) = o01;
    *reinterpret_cast<__nv_bfloat162*>(out + j + 2) = o23;
  }
}

__global__ void __launch_bounds__(kNormThreads) embed_rmsnorm_kernel(const int* tok, const bf16* embed, const bf16* gamma,
                                                                      float eps, int d, int vocab, float* x, bf16* a) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  const int m = blockIdx.x;
  const int t = min(max(tok[m], 0), vocab - 1);  // ids outside the vocabulary read row 0 / V-1
  const bf16* er = embed + static_cast<size_t>(t) * d;
  float* xr = x + static_cast<size_t>(m) * d;
  for (int j = threadIdx.x * 2; j < d; j += blockDim.x * 2) {
    const __nv_bfloat162 e = *reinterpret_cast<const __nv_bfloat162*>(er + j);
    xr[j] = __low2float(e);
    xr[j + 1] = __high2float(e);
  }
  __syncthreads();
  const float inv = row_inv_rms(xr, d, eps, red);
  write_normed(xr, gamma, inv, d, a + static_cast<size_t>(m) * d);
}

// Producer form of the fused RMSNorm: x, bf16(x * gamma) and the row's sum of squares.
__global__ void __launch_bounds__(kNormThreads) embed_scaled_kernel(const int* tok, const bf16* embed, const bf16* gamma,
                                                                    int d, int vocab, float* x, bf16* a, float* ssq) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  const int m = blockIdx.x;
  const int t = min(max(tok[m], 0), vocab - 1);  // ids outside the vocabulary read row 0 / V-1
  const bf16* er = embed + static_cast<size_t>(t) * d;
  float* xr = x + static_cast<size_t>(m) * d;
  bf16* ar = a + static_cast<size_t>(m) * d;
  float ss = 0.f;
  for (int j = threadIdx.x * 2; j < d; j += blockDim.x * 2) {
    const __nv_bfloat162 e = *reinterpret_cast<const __nv_bfloat162*>(er + j);
    const __nv_bfloat162 g = *reinterpret_cast<const __nv_bfloat162*>(gamma + j);
    const float e0 = __low2float(e), e1 = __high2float(e);
    xr[j] = e0;
    xr[j + 1] = e1;
    *reinterpret_cast<__nv_bfloat162*>(ar + j) = __floats2bfloat162_rn(e0 * __low2float(g), e1 * __high2float(g));
    ss += e0 * e0 + e1 * e1;
  }
  ss = block_sum(ss, red);
  if (threadIdx.x == 0) ssq[m] = ss;
}

__global__ void rows_to_bf16_kernel(const float* x, int ld, int w, bf16* out) {
  pdl_trigger();
  pdl_wait();
  const int m = blockIdx.x;
  for (int j = threadIdx.x; j < w; j += blockDim.x)
    out[static_cast<size_t>(m) * w + j] = __float2bfloat16_rn(x[static_cast<size_t>(m) * ld + j]);
}

__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const float* x, const int* rows, const bf16* gamma,
                                                                float eps, int d, bf16* a, float* tap,
                                                                const int* tap_row, int tap_mask) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  const int i = blockIdx.x;
  const int src = rows ? rows[i] : i;
  const float* xr = x + static_cast<size_t>(src) * d;
  const float inv = row_inv_rms(xr, d, eps, red);
  write_normed(xr, gamma, inv, d, a + static_cast<size_t>(i) * d);
  if (tap != nullptr && tap_mask != 0) {
    const int tr = tap_row ? tap_row[src] : src;
    if (tr >= 0) {
      for (int s = 0; s < 3; ++s) {
        if (!(tap_mask & (1 << s))) continue;
        float* dst = tap + (static_cast<size_t>(tr) * 3 + s) * d;
        for (int j = threadIdx.x * 4; j < d; j += blockDim.x * 4)
          *reinterpret_cast<float4*>(dst + j) = *reinterpret_cast<const float4*>(xr + j);
      }
    }
  }
}

// One CTA per row; a work item is 4 consecutive rotation pairs (head, i .. i+3), i < hd/2, over all
// q, k, v heads. The pointers do not alias, and each thread issues the loads of all its items (4 per
// round) before any store, so a row costs about one round trip to L2 instead of one per item.
__global__ void rope_append_kernel(const float* __restrict__ qkv, const float* __restrict__ cs, int H, int Hkv,
                                   int hd, const int* __restrict__ row_seq, const int* __restrict__ row_pos,
                                   const int* __restrict__ row_valid, KVCache kv, int layer, float* __restrict__ q) {
  pdl_trigger();
  pdl_wait();
  constexpr int kPer = 4;
  const int m = blockIdx.x;
  const int half = hd / 2, quads = half / 4;
  const int nh = H + 2 * Hkv, items = nh * quads;
  const int pos = row_pos[m];
  const bool valid = row_valid ? row_valid[m] != 0 : true;
  const float* src = qkv + static_cast<size_t>(m) * nh * hd;
  const float* c = cs + static_cast<size_t>(pos) * half * 2;
  bf16* pool = static_cast<bf16*>(kv.pool);
  size_t blk_base = 0;
  if (valid) {
    const int blk = kv.table[static_cast<size_t>(row_seq[m]) * kv.bt_stride + (pos >> 4)];
    blk_base = (static_cast<size_t>(layer) * kv.n_blocks + blk) * 2 * Hkv * 16 * hd + (pos & 15) * hd;
  }
  for (int base = threadIdx.x; base < items; base += blockDim.x * kPer) {
    float4 x1[kPer], x2[kPer], c0[kPer], c1[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx < items) {
        const int h = idx / quads, i = (idx % quads) * 4;
        x1[u] = *reinterpret_cast<const float4*>(src + h * hd + i);
        x2[u] = *reinterpret_cast<const float4*>(src + h * hd + i + half);
        if (h < H + Hkv) {
          c0[u] = *reinterpret_cast<const float4*>(c + 2 * i);       // cos i, sin i, cos i+1, sin i+1
          c1[u] = *reinterpret_cast<const float4*>(c + 2 * i + 4);   // cos i+2, sin i+2, cos i+3, sin i+3
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx >= items) break;
      const int h = idx / quads, i = (idx % quads) * 4;
      const float4 a = x1[u], b = x2[u];
      if (h < H + Hkv) {
        const float4 r1 = make_float4(a.x * c0[u].x - b.x * c0[u].y, a.y * c0[u].z - b.y * c0[u].w,
                                      a.z * c1[u].x - b.z * c1[u].y, a.w * c1[u].z - b.w * c1[u].w);
        const float4 r2 = make_float4(b.x * c0[u].x + a.x * c0[u].y, b.y * c0[u].z + a.y * c0[u].w,
                                      b.z * c1[u].x + a.z * c1[u].y, b.w * c1[u].z + a.w * c1[u].w);
        if (h < H) {
          float* qo = q + (static_cast<size_t>(m) * H + h) * hd;
          *reinterpret_cast<float4*>(qo + i) = r1;
          *reinterpret_cast<float4*>(qo + i + half) = r2;
        } else if (valid) {
          bf16* ko = pool + blk_base + static_cast<size_t>(h - H) * 16 * hd;
          *reinterpret_cast<uint2*>(ko + i) = make_uint2(pack_bf16x2(r1.x, r1.y), pack_bf16x2(r1.z, r1.w));
          *reinterpret_cast<uint2*>(ko + i + half) = make_uint2(pack_bf16x2(r2.x, r2.y), pack_bf16x2(r2.z, r2.w));
        }
      } else if (valid) {
        bf16* vo = pool + blk_base + static_cast<size_t>(Hkv) * 16 * hd + static_cast<size_t>(h - H - Hkv) * 16 * hd;
        *reinterpret_cast<uint2*>(vo + i) = make_uint2(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w));
        *reinterpret_cast<uint2*>(vo + i + half) = make_uint2(pack_bf16x2(b.x, b.y), pack_bf16x2(b.z, b.w));
      }
    }
  }
}

__global__ void __launch_bounds__(kNormThreads) layernorm_kernel(const float* x, const bf16* gamma, const bf16* beta,
                                                                  float eps, int d, float* g, bf16* g_bf) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  const int b = blockIdx.x;
  const float* xr = x + static_cast<size_t>(b) * d;
  float s = 0.f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) s += xr[j];
  const float mu = block_sum(s, red) / static_cast<float>(d);
  float v = 0.f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float t = xr[j] - mu;
    v += t * t;
  }
  const float var = block_sum(v, red) / static_cast<float>(d);
  const float inv = rsqrtf(var + eps);
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float o = (xr[j] - mu) * inv * bf2f(gamma[j]) + bf2f(beta[j]);
    g[static_cast<size_t>(b) * d + j] = o;
    g_bf[static_cast<size_t>(b) * d + j] = __float2bfloat16_rn(o);
  }
}

__global__ void swiglu_kernel(const float* gate, const float* up, const float* bias, const int* seq, int M, int F,
                              bf16* h) {
  pdl_trigger();
  pdl_wait();
  const size_t n = static_cast<size_t>(M) * F;
  for (size_t idx = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; idx < n;
       idx += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int m = static_cast<int>(idx / F), f = static_cast<int>(idx % F);
    const float g = gate[idx];
    float u = up[idx];
    if (bias) u += bias[static_cast<size_t>(seq ? seq[m] : 0) * F + f];
    h[idx] = __float2bfloat16_rn(u * (g / (1.f + __expf(-g))));
  }
}

__global__ void gather_rows_bf16_kernel(const float* src, int ld_src, const int* idx, int width, bf16* out) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const float* s = src + static_cast<size_t>(b) * ld_src + static_cast<size_t>(idx ? idx[b] : 0) * width;
  for (int j = threadIdx.x; j < width; j += blockDim.x)
    out[static_cast<size_t>(b) * width + j] = __float2bfloat16_rn(s[j]);
}

}  // namespace

cudaError_t embed_rmsnorm(const int* tok, const void* embed, const void* gamma, float eps, int M, int d, int vocab,
                          float* x, void* a, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  { const cudaError_t e_ = launch_pdl(embed_rmsnorm_kernel, dim3(M), dim3(kNormThreads), 0, st, tok, static_cast<const bf16*>(embed),
                                                   static_cast<const bf16*>(gamma), eps, d, vocab, x,
                                                   static_cast<bf16*>(a)); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t embed_scaled(const int* tok, const void* embed, const void* gamma, int M, int d, int vocab, float* x,
                         void* a, float* ssq, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  return launch_pdl(embed_scaled_kernel, dim3(M), dim3(kNormThreads), 0, st, tok, static_cast<const bf16*>(embed),
                    static_cast<const bf16*>(gamma), d, vocab, x, static_cast<bf16*>(a), ssq);
}

cudaError_t rows_to_bf16(const float* x, int ld, int M, int w, void* out, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  return launch_pdl(rows_to_bf16_kernel, dim3(M), dim3(256), 0, st, x, ld, w, static_cast<bf16*>(out));
}

cudaError_t rmsnorm(const float* x, const int* rows, const void* gamma, float eps, int M, int d, void* a, float* tap,
                    const int* tap_row, int tap_mask, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  { const cudaError_t e_ = launch_pdl(rmsnorm_kernel, dim3(M), dim3(kNormThreads), 0, st, x, rows, static_cast<const bf16*>(gamma), eps, d, static_cast<bf16*>(a),
                                             tap, tap_row, tap_mask); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t rope_append(const float* qkv, const float* rope_cs, int M, int H, int Hkv, int hd, const int* row_seq,
                        const int* row_pos, const int* row_valid, const KVCache& kv, int layer, float* q,
                        cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  { const cudaError_t e_ = launch_pdl(rope_append_kernel, dim3(M), dim3(256), 0, st, qkv, rope_cs, H, Hkv, hd, row_seq, row_pos, row_valid, kv, layer, q); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t layernorm(const float* x, const void* gamma, const void* beta, float eps, int B, int d, float* g,
                      void* g_bf, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  { const cudaError_t e_ = launch_pdl(layernorm_kernel, dim3(B), dim3(kNormThreads), 0, st, x, static_cast<const bf16*>(gamma), static_cast<const bf16*>(beta), eps,
                                               d, g, static_cast<bf16*>(g_bf)); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t swiglu(const float* gate, const float* up, const float* bias, const int* seq, int M, int F, void* h,
                   cudaStream_t st) {
  if (M <= 0 || F <= 0) return cudaSuccess;
  const size_t n = static_cast<size_t>(M) * F;
  int blocks = static_cast<int>((n + 255) / 256);
  if (blocks > 152 * 16) blocks = 152 * 16;
  { const cudaError_t e_ = launch_pdl(swiglu_kernel, dim3(blocks), dim3(256), 0, st, gate, up, bias, seq, M, F, static_cast<bf16*>(h)); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t gather_rows_bf16(const float* src, int ld_src, const int* idx, int width, int B, void* out,
                             cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  { const cudaError_t e_ = launch_pdl(gather_rows_bf16_kernel, dim3(B), dim3(256), 0, st, src, ld_src, idx, width, static_cast<bf16*>(out)); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

}  // namespace sd2
