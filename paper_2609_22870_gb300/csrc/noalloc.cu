// fp8rl_token_logprobs_noalloc: the scoring call of fp8rl_token_logprobs for
// callers that cannot hand the library a workspace, because they are not
// allowed to allocate device memory when they call it.  Its scratch (the
// per-token logsumexp partials and the gathered target logits) lives in one
// fixed array compiled into the library instead.
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
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_scratch on the current device.  In host code the name
// g_scratch only stands in for the symbol, so the address comes from the
// runtime, once per device, with that device current.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
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
