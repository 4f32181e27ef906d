// extern "C" entry points of libfp8rl.so (declared in include/fp8rl.h):
// argument validation, workspace carving and kernel dispatch.  No entry point
// allocates device memory; scratch comes from the caller's workspace.
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace fp8rl {

namespace {
constexpr uint64_t kDefaultWaitNs = 2000000000ull;
std::atomic<uint64_t> g_wait_ns{kDefaultWaitNs};
thread_local char g_last_err[256] = "";

fp8rl_status cuda_fail(cudaError_t e) {
  std::snprintf(g_last_err, sizeof(g_last_err), "%s: %s", cudaGetErrorName(e), cudaGetErrorString(e));
  return FP8RL_ECUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool valid_gran(int g) { return g == FP8RL_GRAN_TENSOR || g == FP8RL_GRAN_ROWWISE || g == FP8RL_GRAN_BLOCK; }
// the scoring calls also take the block layout with power-of-two scales
bool valid_score_gran(int g) { return valid_gran(g) || g == FP8RL_GRAN_BLOCK_UE8M0; }
bool block_layout(int g) { return g == FP8RL_GRAN_BLOCK || g == FP8RL_GRAN_BLOCK_UE8M0; }

// Workspace layout of fp8rl_token_logprobs: per-token LSE partials
// [gemm_partials_per_token(V)][T] float2, then z_y [T] float.
size_t partials_bytes(int64_t T, int64_t V) {
  return align_up(static_cast<size_t>(gemm_partials_per_token(V)) * static_cast<size_t>(T) * sizeof(float2), 256);
}
size_t logprob_ws(int64_t T, int64_t V) {
  return partials_bytes(T, V) + align_up(static_cast<size_t>(T) * sizeof(float), 256);
}

fp8rl_status check_gemm_shape(const uint8_t* hc, const float* hs, const uint8_t* wc, const float* wsc,
                              fp8rl_gran g, int64_t T, int64_t H, int64_t V) {
  if (!hc || !hs || !wc || !wsc || !valid_score_gran(g)) return FP8RL_EINVAL;
  if (T < 1 || V < 1 || H < 16) return FP8RL_ESHAPE;
  if (H % 16 != 0 || (block_layout(g) && H % 128 != 0)) return FP8RL_ESHAPE;
  if (T > 0x7FFFFFFF || V > 0x7FFFFFFF || H > 0x7FFFFFFF) return FP8RL_ESHAPE;
  if (!aligned16(hc) || !aligned16(wc)) return FP8RL_EALIGN;
  return FP8RL_OK;
}
}  // namespace

uint64_t wait_limit_ns() { return g_wait_ns.load(std::memory_order_relaxed); }

void record_cuda_error(cudaError_t e) { cuda_fail(e); }

void* tensormap_encoder() {
  static void* fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = ptr;
  }
  return fn;
}

int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) dev = 0;
  if (cached[dev] == 0) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    cached[dev] = n > 0 ? n : 1;
  }
  return cached[dev];
}

int resident_ctas(const void* kernel, int threads) {
  struct Entry {
    int dev;
    const void* fn;
    int threads, n;
  };
  static std::mutex mu;
  static Entry table[64];
  static int used = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (table[i].dev == dev && table[i].fn == kernel && table[i].threads == threads) return table[i].n;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, 0) != cudaSuccess || n < 1) n = 1;
  if (used < 64) table[used++] = Entry{dev, kernel, threads, n};
  return n;
}

}  // namespace fp8rl

using namespace fp8rl;

// Only the entry points declared in fp8rl.h are visible outside the library
// (everything else is compiled with -fvisibility=hidden).
#pragma GCC visibility push(default)
extern "C" {

fp8rl_status fp8rl_check(void* stream) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  uint32_t bits = quantize_status_take() | gemm_status_take() |
                  combine_status_take() | calib_status_take() | loss_status_take();
  if (bits & kErrTimeout) return FP8RL_ETIMEOUT;
  if (bits & kErrDevice) return FP8RL_EDEVICE;
  if (e != cudaSuccess) return cuda_fail(e);
  return FP8RL_OK;
}

const char* fp8rl_status_string(fp8rl_status s) {
  switch (s) {
    case FP8RL_OK: return "ok";
    case FP8RL_EINVAL: return "invalid argument (null pointer or unknown enum)";
    case FP8RL_ESHAPE: return "unsupported shape";
    case FP8RL_EALIGN: return "pointer or leading dimension not 16-byte aligned";
    case FP8RL_EWORKSPACE: return "workspace missing or too small";
    case FP8RL_ECUDA: return "CUDA call failed (see fp8rl_last_cuda_error)";
    case FP8RL_EDEVICE: return "a kernel flagged invalid input data";
    case FP8RL_ETIMEOUT: return "a bounded in-kernel wait expired";
  }
  return "unknown status";
}

const char* fp8rl_last_cuda_error(void) { return g_last_err; }

void fp8rl_set_wait_limit_ns(uint64_t limit_ns) {
  g_wait_ns.store(limit_ns ? limit_ns : kDefaultWaitNs, std::memory_order_relaxed);
}

fp8rl_status fp8rl_wait_selftest(uint64_t limit_ns, void* stream) {
  cudaError_t e = launch_wait_selftest(limit_ns, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

// ------------------------------------------------------------------ quantize
int64_t fp8rl_scales_count(int64_t rows, int64_t cols, fp8rl_gran g, fp8rl_role role) {
  if (rows < 0 || cols < 0 || !valid_score_gran(g)) return 0;
  if (g == FP8RL_GRAN_TENSOR) return 1;
  if (g == FP8RL_GRAN_ROWWISE) return rows;
  if (cols % 128 != 0) return 0;
  if (role == FP8RL_ROLE_ACT) return rows * (cols / 128);
  return (rows + 127) / 128 * (cols / 128);
}

size_t fp8rl_quantize_workspace_size(int64_t, int64_t, fp8rl_gran g, fp8rl_role) {
  return g == FP8RL_GRAN_TENSOR ? 256 : 0;
}

namespace {
fp8rl_status quantize_impl(const void* x, int64_t rows, int64_t cols, int64_t ld, fp8rl_gran g,
                           fp8rl_role role, uint8_t* codes, float* scales, void* ws,
                           size_t ws_bytes, bool pow2, void* stream) {
  if (!x || !codes || !scales || !valid_gran(g)) return FP8RL_EINVAL;
  if (role != FP8RL_ROLE_ACT && role != FP8RL_ROLE_WEIGHT) return FP8RL_EINVAL;
  if (rows < 0 || cols < 16 || ld < cols) return FP8RL_ESHAPE;
  if (cols % 16 != 0 || (g == FP8RL_GRAN_BLOCK && cols % 128 != 0)) return FP8RL_ESHAPE;
  if (!aligned16(x) || !aligned16(codes) || ld % 8 != 0) return FP8RL_EALIGN;
  const size_t need = fp8rl_quantize_workspace_size(rows, cols, g, role);
  if (need && (!ws || ws_bytes < need)) return FP8RL_EWORKSPACE;
  cudaError_t e = launch_quantize(x, rows, cols, ld, g, role, codes, scales, ws, pow2,
                                  static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}
}  // namespace

fp8rl_status fp8rl_quantize(const void* x, int64_t rows, int64_t cols, int64_t ld, fp8rl_gran g,
                            fp8rl_role role, uint8_t* codes, float* scales, void* ws,
                            size_t ws_bytes, void* stream) {
  return quantize_impl(x, rows, cols, ld, g, role, codes, scales, ws, ws_bytes, false, stream);
}

fp8rl_status fp8rl_quantize_ue8m0(const void* x, int64_t rows, int64_t cols, int64_t ld,
                                  fp8rl_gran g, fp8rl_role role, uint8_t* codes, float* scales,
                                  void* ws, size_t ws_bytes, void* stream) {
  return quantize_impl(x, rows, cols, ld, g, role, codes, scales, ws, ws_bytes, true, stream);
}

// ------------------------------------------------------------------ scoring
size_t fp8rl_token_logprobs_workspace_size(int64_t T, int64_t H, int64_t V, fp8rl_gran g) {
  if (T < 0 || V < 0 || H < 0) return 0;
  // the UE8M0 mode adds the scale-factor images of the block-scaled MMA
  return logprob_ws(T, V) + (g == FP8RL_GRAN_BLOCK_UE8M0 ? gemm_ue8m0_image_bytes(T, V, H) : 0);
}

fp8rl_status fp8rl_logit_partials(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                  const float* wsc, fp8rl_gran g, int64_t T, int64_t H, int64_t V,
                                  const int32_t* targets, void* ws, size_t ws_bytes, void* stream) {
  fp8rl_status st = check_gemm_shape(hc, hs, wc, wsc, g, T, H, V);
  if (st != FP8RL_OK) return st;
  if (!targets) return FP8RL_EINVAL;
  if (!ws || ws_bytes < fp8rl_token_logprobs_workspace_size(T, H, V, g)) return FP8RL_EWORKSPACE;
  if (g == FP8RL_GRAN_BLOCK_UE8M0 && !aligned16(ws)) return FP8RL_EALIGN;
  GemmArgs a{};
  a.a_codes = hc;
  a.a_scales = hs;
  a.b_codes = wc;
  a.b_scales = wsc;
  a.gran = g;
  a.M = T;
  a.N = V;
  a.K = H;
  a.targets = targets;
  a.partials = static_cast<float2*>(ws);
  a.zy = reinterpret_cast<float*>(static_cast<char*>(ws) + partials_bytes(T, V));
  if (g == FP8RL_GRAN_BLOCK_UE8M0) a.sf_images = static_cast<uint8_t*>(ws) + logprob_ws(T, V);
  cudaError_t e = launch_gemm_lse(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

fp8rl_status fp8rl_combine_logprobs(int64_t T, int64_t, int64_t V, fp8rl_gran g,
                                    const int32_t* targets, const float* logp_old, float* logp,
                                    float* lse, float* ratio, void* ws, size_t ws_bytes,
                                    void* stream) {
  if (!targets || !logp || !valid_score_gran(g) || (ratio && !logp_old)) return FP8RL_EINVAL;
  if (T < 1 || V < 1) return FP8RL_ESHAPE;
  if (!ws || ws_bytes < logprob_ws(T, V)) return FP8RL_EWORKSPACE;
  const float2* partials = static_cast<const float2*>(ws);
  const float* zy = reinterpret_cast<const float*>(static_cast<const char*>(ws) + partials_bytes(T, V));
  cudaError_t e = launch_combine(partials, zy, targets, logp_old, logp, lse, ratio, T, V,
                                 static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

fp8rl_status fp8rl_token_logprobs(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                  const float* wsc, fp8rl_gran g, int64_t T, int64_t H, int64_t V,
                                  const int32_t* targets, const float* logp_old, float* logp,
                                  float* lse, float* ratio, void* ws, size_t ws_bytes,
                                  void* stream) {
  if (!logp || (ratio && !logp_old)) return FP8RL_EINVAL;
  fp8rl_status st = fp8rl_logit_partials(hc, hs, wc, wsc, g, T, H, V, targets, ws, ws_bytes, stream);
  if (st != FP8RL_OK) return st;
  return fp8rl_combine_logprobs(T, H, V, g, targets, logp_old, logp, lse, ratio, ws, ws_bytes, stream);
}

// ------------------------------------------------------------------ BF16 shadow pass
size_t fp8rl_bf16_token_logprobs_workspace_size(int64_t T, int64_t, int64_t V) {
  if (T < 0 || V < 0) return 0;
  return logprob_ws(T, V);
}

fp8rl_status fp8rl_bf16_token_logprobs(const void* h, int64_t ld_h, const void* w, int64_t ld_w,
                                       int64_t T, int64_t H, int64_t V, const int32_t* targets,
                                       const float* logp_old, float* logp, float* lse, float* ratio,
                                       void* ws, size_t ws_bytes, void* stream) {
  if (!h || !w || !targets || !logp || (ratio && !logp_old)) return FP8RL_EINVAL;
  if (T < 1 || V < 1 || H < 64 || H % 64 != 0 || ld_h < H || ld_w < H) return FP8RL_ESHAPE;
  if (T > 0x7FFFFFFF || V > 0x7FFFFFFF || H > 0x7FFFFFFF) return FP8RL_ESHAPE;
  if (!aligned16(h) || !aligned16(w) || ld_h % 8 != 0 || ld_w % 8 != 0) return FP8RL_EALIGN;
  if (!ws || ws_bytes < logprob_ws(T, V)) return FP8RL_EWORKSPACE;
  GemmArgs a{};
  a.a_codes = h;
  a.b_codes = w;
  a.gran = kGemmBf16;
  a.M = T;
  a.N = V;
  a.K = H;
  a.lda = ld_h;
  a.ldb = ld_w;
  a.targets = targets;
  a.partials = static_cast<float2*>(ws);
  a.zy = reinterpret_cast<float*>(static_cast<char*>(ws) + partials_bytes(T, V));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = launch_gemm_lse(a, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = launch_combine(a.partials, a.zy, targets, logp_old, logp, lse, ratio, T, V, s);
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

fp8rl_status fp8rl_importance_ratios(const float* lp_new, const float* lp_old, int64_t T,
                                     float* ratio, void* stream) {
  if (!lp_new || !lp_old || !ratio) return FP8RL_EINVAL;
  if (T < 0) return FP8RL_ESHAPE;
  cudaError_t e = launch_ratios(lp_new, lp_old, T, ratio, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

// ------------------------------------------------------------------ calibrate
void fp8rl_default_calib_opts(fp8rl_calib_opts* o) {
  if (!o) return;
  o->mode = FP8RL_CALIB_EXACT;
  o->reserved = 0;
  o->lo_min = 0.5;
  o->lo_max = 0.9;
  o->hi_min = 1.2;
  o->hi_max = 2.0;
  o->step = 0.02;
  o->delta_lo = 0.05;
  o->delta_hi = 0.1;
  o->lo_old = NAN;
  o->hi_old = NAN;
}

size_t fp8rl_calibrate_workspace_size(int64_t T) { return T < 0 ? 0 : calib_workspace_bytes(T); }

fp8rl_status fp8rl_calibrate_clip_bounds(const float* r_fp8, const float* r_bf16, const float* adv,
                                         const uint8_t* mask, const float* coef, int64_t T,
                                         float eps_low, float eps_high,
                                         const fp8rl_calib_opts* opts, fp8rl_calib_result* result,
                                         void* ws, size_t ws_bytes, void* stream) {
  if (!result || (T > 0 && (!r_fp8 || !r_bf16 || !adv))) return FP8RL_EINVAL;
  if (T < 0) return FP8RL_ESHAPE;
  fp8rl_calib_opts o;
  if (opts) o = *opts;
  else fp8rl_default_calib_opts(&o);
  if ((o.mode != FP8RL_CALIB_EXACT && o.mode != FP8RL_CALIB_GRID) || o.reserved != 0) return FP8RL_EINVAL;
  if (!std::isfinite(eps_low) || !std::isfinite(eps_high)) return FP8RL_EINVAL;
  if (!(o.lo_min <= o.lo_max) || !(o.hi_min <= o.hi_max) || !(o.delta_lo >= 0) || !(o.delta_hi >= 0) ||
      !(o.lo_min >= 0) || !(o.hi_min >= 0) || !std::isfinite(o.lo_max) || !std::isfinite(o.hi_max))
    return FP8RL_EINVAL;
  if (o.mode == FP8RL_CALIB_GRID) {
    if (!(o.step > 0)) return FP8RL_EINVAL;
    const double nl = std::round((o.lo_max - o.lo_min) / o.step) + 1;
    const double nh = std::round((o.hi_max - o.hi_min) / o.step) + 1;
    if (nl > 2047 || nh > 2047) return FP8RL_ESHAPE;
  }
  if (!ws || ws_bytes < calib_workspace_bytes(T)) return FP8RL_EWORKSPACE;
  cudaError_t e = launch_calibrate(r_fp8, r_bf16, adv, mask, coef, T, eps_low, eps_high, o, result,
                                   ws, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

// ------------------------------------------------------------------ surrogate
size_t fp8rl_surrogate_workspace_size(int64_t T) { return T < 0 ? 0 : surrogate_workspace_bytes(T); }

fp8rl_status fp8rl_clipped_surrogate(const float* r, const float* adv, const uint8_t* mask,
                                     const float* w_tis, int64_t T, float lo, float hi,
                                     const float* bounds, const int64_t* n_valid, float* grad,
                                     uint8_t* clip_mask, fp8rl_clip_stats* stats, void* ws,
                                     size_t ws_bytes, void* stream) {
  if (!stats || (T > 0 && (!r || !adv))) return FP8RL_EINVAL;
  if (T < 0) return FP8RL_ESHAPE;
  if (!ws || ws_bytes < surrogate_workspace_bytes(T)) return FP8RL_EWORKSPACE;
  cudaError_t e = launch_surrogate(r, adv, mask, w_tis, T, lo, hi, bounds, n_valid, grad, clip_mask,
                                   stats, ws, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

size_t fp8rl_surrogate_seq_mean_workspace_size(int64_t T, int64_t n_seq) {
  return (T < 0 || n_seq < 0) ? 0 : seq_surrogate_workspace_bytes(T, n_seq);
}

fp8rl_status fp8rl_clipped_surrogate_seq_mean(const float* r, const float* adv, const uint8_t* mask,
                                              const float* w_tis, const int32_t* seq_id,
                                              int64_t n_seq, int64_t T, float lo, float hi,
                                              const float* bounds, float* grad, uint8_t* clip_mask,
                                              fp8rl_clip_stats* stats, void* ws, size_t ws_bytes,
                                              void* stream) {
  if (!stats || (T > 0 && (!r || !adv || !seq_id))) return FP8RL_EINVAL;
  if (T < 0 || n_seq < 0 || n_seq > 0x7FFFFFFF) return FP8RL_ESHAPE;
  if (!ws || ws_bytes < seq_surrogate_workspace_bytes(T, n_seq)) return FP8RL_EWORKSPACE;
  cudaError_t e = launch_seq_surrogate(r, adv, mask, w_tis, seq_id, n_seq, T, lo, hi, bounds, grad,
                                       clip_mask, stats, ws, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

size_t fp8rl_seq_level_surrogate_workspace_size(int64_t T, int64_t n_seq) {
  return (T < 0 || n_seq < 0) ? 0 : seq_level_workspace_bytes(T, n_seq);
}

fp8rl_status fp8rl_seq_level_clipped_surrogate(const float* logp, const float* logp_old,
                                               const float* adv_seq, const uint8_t* mask,
                                               const int32_t* seq_id, int64_t n_seq, int64_t T,
                                               float lo, float hi, const float* bounds,
                                               float* seq_ratio, uint8_t* seq_clip, float* grad,
                                               fp8rl_clip_stats* stats, void* ws, size_t ws_bytes,
                                               void* stream) {
  if (!stats || (T > 0 && (!logp || !logp_old || !seq_id)) || (n_seq > 0 && !adv_seq))
    return FP8RL_EINVAL;
  if (T < 0 || n_seq < 0 || n_seq > 0x7FFFFFFF) return FP8RL_ESHAPE;
  if (!ws || ws_bytes < seq_level_workspace_bytes(T, n_seq)) return FP8RL_EWORKSPACE;
  cudaError_t e = launch_seq_level(logp, logp_old, adv_seq, mask, seq_id, n_seq, T, lo, hi, bounds,
                                   seq_ratio, seq_clip, grad, stats, ws,
                                   static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

// ------------------------------------------------------------------ diagnostics
size_t fp8rl_clip_diagnostics_workspace_size(int64_t T) { return T < 0 ? 0 : diag_workspace_bytes(T); }

fp8rl_status fp8rl_clip_diagnostics(const float* lp8, const float* lpb, const float* r8,
                                    const float* rb, const float* adv, const uint8_t* mask,
                                    int64_t T, float eps_low, float eps_high, fp8rl_clip_diag* out,
                                    void* ws, size_t ws_bytes, void* stream) {
  if (!out || (T > 0 && (!r8 || !rb || !adv)) || ((lp8 == nullptr) != (lpb == nullptr)))
    return FP8RL_EINVAL;
  if (!std::isfinite(eps_low) || !std::isfinite(eps_high)) return FP8RL_EINVAL;
  if (T < 0) return FP8RL_ESHAPE;
  if (!ws || ws_bytes < diag_workspace_bytes(T)) return FP8RL_EWORKSPACE;
  cudaError_t e = launch_clip_diag(lp8, lpb, r8, rb, adv, mask, T, 1.0f - eps_low, 1.0f + eps_high,
                                   out, ws, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

fp8rl_status fp8rl_tis_weights(const float* lp_old, const float* lp_samp, int64_t T, float C,
                               float* w, void* stream) {
  if (T > 0 && (!lp_old || !lp_samp || !w)) return FP8RL_EINVAL;
  if (!std::isfinite(C) || !(C > 0.f)) return FP8RL_EINVAL;
  if (T < 0) return FP8RL_ESHAPE;
  cudaError_t e = launch_tis(lp_old, lp_samp, T, C, w, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

// ------------------------------------------------------------------ dlogits
// Workspace: gathered codes [n][H], scales, targets, lse, grad.
static size_t dl_codes_bytes(int64_t n, int64_t H) { return align_up(static_cast<size_t>(n * H), 256); }
static size_t dl_scales_bytes(int64_t n, int64_t H) {
  return align_up(static_cast<size_t>((n > 0 ? n : 1) * (H / 128 > 0 ? H / 128 : 1)) * 4 + 4, 256);
}
static size_t dl_vec_bytes(int64_t n) { return align_up(static_cast<size_t>(n > 0 ? n : 1) * 4, 256); }

size_t fp8rl_dlogits_workspace_size(int64_t n, int64_t H, int64_t V, fp8rl_gran g) {
  if (n < 0 || H < 0 || V < 0) return 0;
  return dl_codes_bytes(n, H) + dl_scales_bytes(n, H) + 3 * dl_vec_bytes(n) +
         (g == FP8RL_GRAN_BLOCK_UE8M0 ? gemm_ue8m0_image_bytes(n, V, H) : 0);
}

fp8rl_status fp8rl_dlogits_rows(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                const float* wsc, fp8rl_gran g, int64_t T, int64_t H, int64_t V,
                                const int32_t* targets, const float* lse, const float* grad,
                                const int64_t* rows, int64_t n_rows, float* out, void* ws,
                                size_t ws_bytes, void* stream) {
  fp8rl_status st = check_gemm_shape(hc, hs, wc, wsc, g, T, H, V);
  if (st != FP8RL_OK) return st;
  if (!targets || !lse || !grad || (n_rows > 0 && (!rows || !out))) return FP8RL_EINVAL;
  if (n_rows < 0 || n_rows > 0x7FFFFFFF) return FP8RL_ESHAPE;
  if (n_rows == 0) return FP8RL_OK;
  if (!ws || ws_bytes < fp8rl_dlogits_workspace_size(n_rows, H, V, g)) return FP8RL_EWORKSPACE;
  if (!aligned16(ws)) return FP8RL_EALIGN;
  char* p = static_cast<char*>(ws);
  uint8_t* g_codes = reinterpret_cast<uint8_t*>(p);
  p += dl_codes_bytes(n_rows, H);
  float* g_scales = reinterpret_cast<float*>(p);
  p += dl_scales_bytes(n_rows, H);
  int32_t* g_t = reinterpret_cast<int32_t*>(p);
  p += dl_vec_bytes(n_rows);
  float* g_lse = reinterpret_cast<float*>(p);
  p += dl_vec_bytes(n_rows);
  float* g_grad = reinterpret_cast<float*>(p);
  p += dl_vec_bytes(n_rows);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = launch_gather_rows(hc, hs, g, T, H, targets, lse, grad, rows, n_rows, g_codes,
                                     g_scales, g_t, g_lse, g_grad, s);
  if (e != cudaSuccess) return cuda_fail(e);
  GemmArgs a{};
  a.a_codes = g_codes;
  a.a_scales = g_scales;
  a.b_codes = wc;
  a.b_scales = wsc;
  a.gran = g;
  a.M = n_rows;
  a.N = V;
  a.K = H;
  a.targets = g_t;
  a.lse = g_lse;
  a.grad = g_grad;
  a.out = out;
  if (g == FP8RL_GRAN_BLOCK_UE8M0) a.sf_images = reinterpret_cast<uint8_t*>(p);
  e = launch_gemm_dlogits(a, s);
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

// ------------------------------------------------------------------ lm_head backward
// The GEMMs index rows and K with 32-bit ints: T and V (and their 128-padded
// K extents) must stay below 2^31.
constexpr int64_t kMaxBwdRows = (int64_t{1} << 31) - 256;

size_t fp8rl_lm_head_backward_workspace_size(int64_t T, int64_t H, int64_t V) {
  return (T < 1 || H < 1 || V < 1) ? 0 : bwd_layout(T, H, V).total;
}

fp8rl_status fp8rl_lm_head_backward(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                    const float* wsc, fp8rl_gran g, int64_t T, int64_t H, int64_t V,
                                    const int32_t* targets, const float* lse, const float* grad,
                                    const void* h_bf16, const void* w_bf16, float* dh, float* dW,
                                    int flags, void* ws, size_t ws_bytes, void* stream) {
  fp8rl_status st = check_gemm_shape(hc, hs, wc, wsc, g, T, H, V);
  if (st != FP8RL_OK) return st;
  if (!targets || !lse || !grad || !h_bf16 || !w_bf16 || (!dh && !dW)) return FP8RL_EINVAL;
  if (flags & ~(FP8RL_BWD_ACCUMULATE_DW | FP8RL_BWD_POW2_SCALES)) return FP8RL_EINVAL;
  if (T > kMaxBwdRows || V > kMaxBwdRows) return FP8RL_ESHAPE;
  if (!aligned16(h_bf16) || !aligned16(w_bf16) || (dh && !aligned16(dh)) || (dW && !aligned16(dW)))
    return FP8RL_EALIGN;
  if (!ws || ws_bytes < bwd_layout(T, H, V).total) return FP8RL_EWORKSPACE;
  if (!aligned16(ws)) return FP8RL_EALIGN;
  cudaError_t e = launch_lm_head_backward(hc, hs, wc, wsc, g, T, H, V, targets, lse, grad,
                                          static_cast<const uint16_t*>(h_bf16),
                                          static_cast<const uint16_t*>(w_bf16), dh, dW,
                                          (flags & FP8RL_BWD_ACCUMULATE_DW) != 0,
                                          (flags & FP8RL_BWD_POW2_SCALES) != 0,
                                          ws, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FP8RL_OK : cuda_fail(e);
}

}  // extern "C"
#pragma GCC visibility pop
