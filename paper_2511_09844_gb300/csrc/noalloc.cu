// sd2_accept_logits_noalloc: the speculative acceptance of sd2_accept_logits for callers that
// cannot allocate device memory at all.
//
// Who needs it: code that runs inside a host process whose device memory belongs to somebody
// else's allocator (a plugin inside an inference server or framework that hands out no
// allocator handle), and loops that must not call cudaMalloc/cudaFree because those calls can
// synchronise the whole device at a point the caller does not control. Such callers can pass
// their logits and outputs but cannot provide the workspace that sd2_accept_logits asks for.
//
// So this variant keeps its workspace in a fixed, file-scope device array that every GPU which
// loads the library holds until the process exits. Its size is kScratchBytes (256 KiB). The
// acceptance tables sit at its start and take 16*B*(2k+1) + 28*B + 64 bytes; the last
// kErrBytes hold the error word that sd2_accept_logits_noalloc_check reads back. A request
// whose tables would reach the error word (more than 261888 bytes; B = 256 with k = 16 needs
// 142400) is rejected with SD2_ECAPACITY. Nothing here calls cudaMalloc, cudaFree or any
// allocating routine.
#include <cuda.h>

#include <mutex>
#include <string>

#include "sd2.h"
#include "common.cuh"
#include "kernels.h"

namespace sd2 {
void record_last_error(const std::string& m);  // engine.cu
}

namespace {

constexpr size_t kScratchBytes = 256 * 1024;
constexpr size_t kErrBytes = 256;                      // the error word's slot at the end of the array
constexpr size_t kTableBytes = kScratchBytes - kErrBytes;
constexpr int kMaxContexts = 64;

// The shared workspace. In host code this name is only a stand-in for the device symbol: its
// device address must come from cudaGetSymbolAddress in the caller's context, never from &scratch.
static __device__ __align__(256) unsigned char scratch[kScratchBytes];

// Device addresses of `scratch`, one per CUDA context that has called in. A __device__ symbol's
// address belongs to a context (the device's primary context, or one the caller created and made
// current), so the cache is keyed on the context's unique id, which CUDA never reuses within a
// process (a context recreated after cudaDeviceReset gets a new id and a fresh lookup).
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);
std::mutex g_mu;
unsigned long long g_ctx_id[kMaxContexts] = {};
void* g_ctx_ptr[kMaxContexts] = {};
int g_n_ctx = 0, g_next_slot = 0;

// Errors are reported like every context-free call: the status here, the text through
// sd2_last_error(NULL).
sd2_status fail(sd2_status s, const std::string& m) {
  sd2::record_last_error(m);
  return s;
}

bool driver_fns(CtxGetCurrentFn* cur, CtxGetIdFn* id) {
  static CtxGetCurrentFn f_cur = nullptr;
  static CtxGetIdFn f_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f_cur = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  *cur = f_cur;
  *id = f_id;
  return f_cur && f_id;
}

// Id of the current context, or 0 when none is current yet.
unsigned long long current_ctx_id(CtxGetCurrentFn cur, CtxGetIdFn id) {
  CUcontext ctx = nullptr;
  unsigned long long v = 0;
  if (cur(&ctx) != CUDA_SUCCESS || !ctx) return 0;
  if (id(ctx, &v) != CUDA_SUCCESS) return 0;
  return v;
}

// Device address of `scratch` in the current context: looked up once per context (the lookup
// also brings up the runtime's context when none is current yet), then served from the table.
sd2_status scratch_address(void** out) {
  CtxGetCurrentFn cur;
  CtxGetIdFn id;
  if (!driver_fns(&cur, &id)) return fail(SD2_ECUDA, "cuCtxGetCurrent/cuCtxGetId unavailable from the driver");
  std::lock_guard<std::mutex> lock(g_mu);
  unsigned long long cid = current_ctx_id(cur, id);
  for (int i = 0; cid && i < g_n_ctx; ++i)
    if (g_ctx_id[i] == cid) {
      *out = g_ctx_ptr[i];
      return SD2_OK;
    }
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, scratch);
  if (e != cudaSuccess || p == nullptr)
    return fail(SD2_ECUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
  if (!cid) cid = current_ctx_id(cur, id);
  if (cid) {   // remember it (the oldest entry makes room once the table is full)
    const int slot = g_n_ctx < kMaxContexts ? g_n_ctx++ : (g_next_slot++ % kMaxContexts);
    g_ctx_id[slot] = cid;
    g_ctx_ptr[slot] = p;
  }
  *out = p;
  return SD2_OK;
}

}  // namespace

extern "C" {

sd2_status sd2_accept_logits_noalloc(const void* d_target, const void* d_draft, int32_t dtype, const int32_t* d_xhat,
                                     const float* d_temperature, int32_t B, int32_t k, int32_t V, uint64_t seed,
                                     uint32_t step, int32_t* d_tokens, int32_t* d_n, void* stream) {
  if (!d_target || !d_draft || !d_xhat || !d_temperature || !d_tokens || !d_n)
    return fail(SD2_EINVAL, "null argument");
  if (dtype != SD2_DTYPE_F32 && dtype != SD2_DTYPE_BF16) return fail(SD2_EINVAL, "dtype must be F32 or BF16");
  if (B < 1 || k < 1 || k > 64 || V < 4 || V % 4) return fail(SD2_EINVAL, "need B >= 1, 1 <= k <= 64, V % 4 == 0");
  const size_t align = dtype == SD2_DTYPE_F32 ? 16 : 8;
  if ((reinterpret_cast<uintptr_t>(d_target) | reinterpret_cast<uintptr_t>(d_draft)) & (align - 1))
    return fail(SD2_EINVAL, "logits not aligned for vector loads");
  const size_t need = sd2::accept_scratch_bytes(B, k);
  if (need > kTableBytes)
    return fail(SD2_ECAPACITY, "B*(2k+1) = " + std::to_string(static_cast<long long>(B) * (2 * k + 1)) +
                                   " rows need " + std::to_string(need) + " scratch bytes; the fixed scratch holds " +
                                   std::to_string(kTableBytes) + " for the tables");
  void* base = nullptr;
  sd2_status s = scratch_address(&base);
  if (s != SD2_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  sd2::AcceptScratch sc = sd2::accept_scratch_carve(base, B, k);
  unsigned* err = reinterpret_cast<unsigned*>(static_cast<unsigned char*>(base) + kTableBytes);
  // What must start at zero: the error word here; the row tables are cleared and the race slots
  // and counters reset inside accept_blocks before they are used.
  cudaError_t e = cudaMemsetAsync(err, 0, sizeof(unsigned), st);
  if (e == cudaSuccess)
    e = sd2::accept_blocks(d_target, d_draft, dtype, d_xhat, d_temperature, B, k, V, sd2::Seed{seed, nullptr}, step, nullptr, nullptr,
                           d_tokens, d_n, sc, err, st);
  if (e != cudaSuccess) return fail(SD2_ECUDA, std::string("acceptance launch: ") + cudaGetErrorString(e));
  return SD2_OK;
}

sd2_status sd2_accept_logits_noalloc_check(void* stream) {
  void* base = nullptr;
  sd2_status s = scratch_address(&base);
  if (s != SD2_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  unsigned w = 0;
  cudaError_t e = cudaStreamSynchronize(st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(&w, static_cast<unsigned char*>(base) + kTableBytes, sizeof(unsigned), cudaMemcpyDeviceToHost,
                        st);
  if (e == cudaSuccess) e = cudaMemsetAsync(static_cast<unsigned char*>(base) + kTableBytes, 0, sizeof(unsigned), st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail(SD2_ECUDA, std::string("reading the acceptance error word: ") + cudaGetErrorString(e));
  if (w & sd2::ERR_NONFINITE) return fail(SD2_ENUMERIC, "non-finite logits seen by the last acceptance call");
  if (w & sd2::ERR_TIMEOUT) return fail(SD2_ETIMEOUT, "a device-side wait of the last acceptance call timed out");
  return SD2_OK;
}

}  // extern "C"
