// Row-wise decoder kernels: embedding + RMSNorm, RMSNorm with hidden-state taps, rotary
// embedding with the paged KV append, the steering vector's layer norm (App. A.2), the steered
// SwiGLU of Eq. 2 on precomputed projections, and the f32 -> bf16 row gather of the taps.
#include "common.cuh"
#include "kernels.h"

namespace sd2 {
namespace {

constexpr int kNormThreads = 256;

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

// One CTA per row; thread t handles rotation pairs (head, i) with i < hd/2 over all q, k, v heads.
__global__ void rope_append_kernel(const float* qkv, const float* cs, int H, int Hkv, int hd, const int* row_seq,
                                   const int* row_pos, const int* row_valid, KVCache kv, int layer, float* q) {
  pdl_trigger();
  pdl_wait();
  const int m = blockIdx.x;
  const int half = hd / 2;
  const int nh = H + 2 * Hkv;
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
  for (int idx = threadIdx.x; idx < nh * half; idx += blockDim.x) {
    const int h = idx / half, i = idx % half;
    const float x1 = src[h * hd + i], x2 = src[h * hd + i + half];
    if (h < H + Hkv) {
      const float cv = c[2 * i], sv = c[2 * i + 1];
      const float r1 = x1 * cv - x2 * sv, r2 = x2 * cv + x1 * sv;
      if (h < H) {
        float* qo = q + (static_cast<size_t>(m) * H + h) * hd;
        qo[i] = r1;
        qo[i + half] = r2;
      } else if (valid) {
        bf16* ko = pool + blk_base + static_cast<size_t>(h - H) * 16 * hd;
        ko[i] = __float2bfloat16_rn(r1);
        ko[i + half] = __float2bfloat16_rn(r2);
      }
    } else if (valid) {
      bf16* vo = pool + blk_base + static_cast<size_t>(Hkv) * 16 * hd + static_cast<size_t>(h - H - Hkv) * 16 * hd;
      vo[i] = __float2bfloat16_rn(x1);
      vo[i + half] = __float2bfloat16_rn(x2);
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
