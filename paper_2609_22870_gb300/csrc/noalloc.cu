// fp8rl_token_logprobs_noalloc: the scoring call of fp8rl_token_logprobs for
// callers that may not allocate device memory when they score tokens (serving
// loops and other hot paths that forbid allocation and the device-wide
// synchronisation cudaMalloc / cudaFree can cause, or processes whose device
// memory is all reserved up front), so they cannot hand the library a
// workspace.  Its scratch (the per-token logsumexp partials and the gathered
// target logits) lives in one fixed array compiled into the library instead.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "internal.h"

namespace fp8rl {
namespace {

// Scratch shared by every call on a device.  It is part of the library image:
// each GPU that loads libfp8rl.so holds these 16 MiB until the process exits.
constexpr size_t kScratchBytes = FP8RL_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
struct Cached {
  unsigned long long ctx_id;  // 0 = nothing cached
  void* ptr;
};
Cached g_cache[kMaxDevices] = {};

// Unique id of the context current on this thread (0 if none or if the driver
// lacks the query).  Ids are never reused within a process, so a context
// created after cudaDeviceReset gets a new one.
unsigned long long current_context_id() {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(f);
  });
  if (get_current == nullptr || get_id == nullptr) return 0;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
  unsigned long long id = 0;
  return get_id(ctx, &id) == CUDA_SUCCESS ? id : 0;
}

// Device address of g_scratch on the current device.  In host code the name
// g_scratch only stands in for the symbol, so the address comes from the
// runtime (cudaGetSymbolAddress) with that device current.  It is looked up
// once per device context and again whenever the context changes (after
// cudaDeviceReset the module is loaded anew and the old address is stale).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mutex);
  const unsigned long long id = current_context_id();
  if (id != 0 && g_cache[dev].ctx_id == id) {
    *out = g_cache[dev].ptr;
    return cudaSuccess;
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_scratch);
  if (e != cudaSuccess) return e;
  // the lookup above made the device's primary context current if it was not
  g_cache[dev].ctx_id = id != 0 ? id : current_context_id();
  g_cache[dev].ptr = p;
  *out = p;
  return cudaSuccess;
}

}  // namespace
}  // namespace fp8rl

using namespace fp8rl;

extern "C" __attribute__((visibility("default"))) fp8rl_status fp8rl_token_logprobs_noalloc(
    const uint8_t* h_codes, const float* h_scales, const uint8_t* w_codes, const float* w_scales,
    fp8rl_gran gran, int64_t T, int64_t H, int64_t V, const int32_t* targets,
    const float* logp_old, float* logp, float* lse, float* ratio, void* stream) {
  if (T < 0 || V < 0) return FP8RL_ESHAPE;
  // Refuse shapes whose scratch would not fit the fixed array.
  const size_t need = fp8rl_token_logprobs_workspace_size(T, H, V, gran);
  if (need > kScratchBytes) return FP8RL_EWORKSPACE;
  void* scratch = nullptr;
  const cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) {
    record_cuda_error(e);
    return FP8RL_ECUDA;
  }
  // The GEMM rewrites every partial and z_y that the combine reads, so no part
  // of the scratch has to start at zero.
  return fp8rl_token_logprobs(h_codes, h_scales, w_codes, w_scales, gran, T, H, V, targets, logp_old,
                              logp, lse, ratio, scratch, kScratchBytes, stream);
}
