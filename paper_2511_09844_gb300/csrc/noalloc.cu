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
// loads the library holds until the process exits. Its size is kScratchBytes (256 KiB); the
// acceptance tables take 16*B*(2k+1) + 28*B + 68 bytes (B = 256 with k = 16: 142404 bytes), and
// larger requests are rejected with SD2_ECAPACITY. Nothing here calls cudaMalloc, cudaFree or any
// allocating routine.
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
constexpr int kMaxDevices = 64;

// The shared workspace. In host code this name is only a stand-in for the device symbol: its
// device address must come from cudaGetSymbolAddress on each device, never from &scratch.
static __device__ __align__(256) unsigned char scratch[kScratchBytes];

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Errors are reported like every context-free call: the status here, the text through
// sd2_last_error(NULL).
sd2_status fail(sd2_status s, const std::string& m) {
  sd2::record_last_error(m);
  return s;
}

// Device address of `scratch` on the current device, looked up once per device.
sd2_status scratch_address(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(SD2_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(SD2_EINVAL, "device index out of range for the scratch table");
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, scratch);
    if (e != cudaSuccess || p == nullptr)
      return fail(SD2_ECUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
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
  const size_t need = sd2::accept_scratch_bytes(B, k) + sizeof(unsigned);
  if (need > kScratchBytes)
    return fail(SD2_ECAPACITY, "B*(2k+1) = " + std::to_string(static_cast<long long>(B) * (2 * k + 1)) +
                                   " rows need " + std::to_string(need) + " scratch bytes; the fixed scratch holds " +
                                   std::to_string(kScratchBytes));
  void* base = nullptr;
  sd2_status s = scratch_address(&base);
  if (s != SD2_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  sd2::AcceptScratch sc = sd2::accept_scratch_carve(base, B, k);
  unsigned* err = reinterpret_cast<unsigned*>(sc.jmode + 2 * B);
  // What must start at zero: the error word here; the row tables are cleared and the race slots
  // and counters reset inside accept_blocks before they are used.
  cudaError_t e = cudaMemsetAsync(err, 0, sizeof(unsigned), st);
  if (e == cudaSuccess)
    e = sd2::accept_blocks(d_target, d_draft, dtype, d_xhat, d_temperature, B, k, V, seed, step, nullptr, nullptr,
                           d_tokens, d_n, sc, err, st);
  if (e != cudaSuccess) return fail(SD2_ECUDA, std::string("acceptance launch: ") + cudaGetErrorString(e));
  return SD2_OK;
}

}  // extern "C"
