// Device-resident bookkeeping of the draft-and-verify loop: the row plans of each forward pass
// (token, position, sequence, validity per row), the commit that appends accepted tokens and
// rolls both KV caches back, and the prefill initialisation. Every length lives on the device,
// so a whole iteration can be replayed from a CUDA graph without a host round trip.
//
// Per sequence b with n committed tokens (state rows: n, drafter cached length D, last j, stopped):
//   drafter step 1   rows 2b, 2b+1 = the pending tokens at positions D..n-1 (D = n-1 or n-2);
//                    when only one is pending, row 2b repeats row 2b+1 and writes no KV
//   drafter step i   row b = draft i-1 at position n+i-2
//   verifier         rows b(k+1)+t = [x_{n-1}, draft 1..k] at positions n-1+t
//   commit (j kept)  n += j+1; D = min(n_old + j, n_old + k - 1); verifier cache = n-1 positions
//                    implicitly (it only ever reads positions below each row's own).
#include "common.cuh"
#include "kernels.h"
#include "state.h"
#include "tc.cuh"

namespace sd2 {
namespace {

__device__ __forceinline__ void put(int* tok, int* pos, int* seq, int* valid, int r, int t, int p, int s, int v) {
  tok[r] = t; pos[r] = p; seq[r] = s; valid[r] = v;
}

__global__ void plan_kernel(int mode, int i, int B, int k, int max_ctx, const int* state, int maxB,
                            const int* committed, const int* xhat, int* tok, int* pos, int* seq, int* valid) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int n = state[b], D = state[maxB + b], stop = state[3 * maxB + b];
  const int* cb = committed + static_cast<size_t>(b) * max_ctx;
  const int live = stop ? 0 : 1;
  const int cap = max_ctx - 1;
  if (mode == PLAN_DRAFT_FIRST) {
    const int last = cb[n - 1];
    if (n - D == 2) put(tok, pos, seq, valid, 2 * b, cb[n - 2], min(n - 2, cap), b, live);
    else put(tok, pos, seq, valid, 2 * b, last, min(n - 1, cap), b, 0);
    put(tok, pos, seq, valid, 2 * b + 1, last, min(n - 1, cap), b, live);
  } else if (mode == PLAN_DRAFT_NEXT) {
    put(tok, pos, seq, valid, b, xhat[b * k + i - 2], min(n + i - 2, cap), b, live);
  } else {
    for (int t = 0; t <= k; ++t) {
      const int tk = t == 0 ? cb[n - 1] : xhat[b * k + t - 1];
      put(tok, pos, seq, valid, b * (k + 1) + t, tk, min(n - 1 + t, cap), b, live);
    }
  }
}

__global__ void commit_kernel(int B, int k, int max_ctx, int* state, int maxB, int* committed, const int* tokens,
                              const int* n_out, int* iter) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b == 0) *iter += 1;
  if (b >= B) return;
  if (state[3 * maxB + b]) return;
  const int ne = n_out[b];
  const int j = ne - 1;
  const int n0 = state[b];
  int* cb = committed + static_cast<size_t>(b) * max_ctx;
  for (int t = 0; t < ne; ++t) cb[n0 + t] = tokens[b * (k + 1) + t];
  state[maxB + b] = min(n0 + j, n0 + k - 1);
  state[b] = n0 + ne;
  state[2 * maxB + b] = j;
  if (n0 + ne + k + 1 > max_ctx) state[3 * maxB + b] = 1;
}

// After the prefill sample: committed[b] = prompt + first token; n = len+1, D = len, j = 0.
__global__ void prefill_init_kernel(int B, int max_ctx, const int* prompts, const int* cu, const int* first,
                                    int* state, int maxB, int* committed, int* first_out) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int off = cu[b], len = cu[b + 1] - cu[b];
  int* cb = committed + static_cast<size_t>(b) * max_ctx;
  for (int t = threadIdx.x; t < len; t += blockDim.x) cb[t] = prompts[off + t];
  if (threadIdx.x == 0) {
    cb[len] = first[b];
    if (first_out) first_out[b] = first[b];
    state[b] = len + 1;
    state[maxB + b] = len;
    state[2 * maxB + b] = 0;
    state[3 * maxB + b] = 0;
  }
}

// One bounded mbarrier wait, in the form every wait of the library's kernels takes
// (tc::wait_bar_limit), on a barrier that nothing arrives on: after `cycles` clock cycles the wait
// gives up, latches ERR_TIMEOUT in *err and the kernel returns. Nothing is in flight when it does.
__global__ void expire_wait_kernel(unsigned* err, long long cycles) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(tc::smem_u32(&bar), 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) tc::wait_bar_limit(tc::smem_u32(&bar), 0, &abort_flag, err, cycles);
}

}  // namespace

cudaError_t expire_wait(unsigned* err, long long cycles, cudaStream_t st) {
  expire_wait_kernel<<<1, 32, 0, st>>>(err, cycles);
  return cudaGetLastError();
}

cudaError_t plan_rows(int mode, int i, int B, int k, int max_ctx, const int* state, int maxB, const int* committed,
                      const int* xhat, int* tok, int* pos, int* seq, int* valid, cudaStream_t st) {
  { const cudaError_t e_ = launch_pdl(plan_kernel, dim3((B + 127) / 128), dim3(128), 0, st, mode, i, B, k, max_ctx, state, maxB, committed, xhat, tok, pos, seq,
                                                valid); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t commit(int B, int k, int max_ctx, int* state, int maxB, int* committed, const int* tokens, const int* n_out,
                   int* iter, cudaStream_t st) {
  { const cudaError_t e_ = launch_pdl(commit_kernel, dim3((B + 127) / 128), dim3(128), 0, st, B, k, max_ctx, state, maxB, committed, tokens, n_out, iter); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

cudaError_t prefill_init(int B, int max_ctx, const int* prompts, const int* cu, const int* first, int* state, int maxB,
                         int* committed, int* first_out, cudaStream_t st) {
  { const cudaError_t e_ = launch_pdl(prefill_init_kernel, dim3(B), dim3(256), 0, st, B, max_ctx, prompts, cu, first, state, maxB, committed, first_out); if (e_ != cudaSuccess) return e_; }
  return cudaGetLastError();
}

}  // namespace sd2
