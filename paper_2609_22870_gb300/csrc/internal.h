// Host-side interface between the C ABI (api.cu) and the kernel translation
// units.  Nothing here is exported from libfp8rl.so.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "fp8rl.h"

namespace fp8rl {

// Bounded-wait limit for every in-kernel spin-wait (nanoseconds of GPU time).
uint64_t wait_limit_ns();

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ------------------------------------------------------------- quantize.cu
cudaError_t launch_quantize(const void* x, int64_t rows, int64_t cols, int64_t ld, int gran,
                            int role, uint8_t* codes, float* scales, void* ws, bool pow2,
                            cudaStream_t s);
uint32_t quantize_status_take();

// ----------------------------------------------------------------- gemm.cu
struct GemmArgs {
  const void* a_codes;      // [M][K] E4M3 codes, or bf16 values when gran == kGemmBf16
  const float* a_scales;
  const void* b_codes;      // [N][K]
  const float* b_scales;
  int gran;                 // fp8rl_gran, or kGemmBf16 (BF16 shadow pass, no scales)
  int64_t M, N, K;
  int64_t lda, ldb;         // row strides in elements (0 = K)
  const int32_t* targets;   // [M]
  // LSE epilogue outputs (workspace)
  float2* partials;         // [gemm_partials_per_token(N)][M]
  float* zy;                // [M]
  // dlogits epilogue
  const float* lse;         // [M]
  const float* grad;        // [M]
  float* out;               // [M][N]
  // dense dlogits epilogue (E4M3 codes and scales, both orientations)
  uint8_t* pq_out;          // [M][ld_pq], 1x128 blocks along N
  float* pq_scales;         // [ld_pq / 128][M]
  uint8_t* ptq_out;         // [N][ld_ptq], 128 x 128 blocks
  float* ptq_scales;        // [ld_ptq / 128][N]
  int64_t ld_pq, ld_ptq;
  // store epilogue (fp32 accumulators)
  float* c_out;             // [M][ld_c], 16-byte aligned, ld_c % 4 == 0
  int64_t ld_c;
  int accumulate;           // add to c_out instead of overwriting it
  int p_pow2;               // dense FP8 dlogits: power-of-two scales for P and P^T
  // FP8RL_GRAN_BLOCK_UE8M0: device scratch of gemm_ue8m0_image_bytes(M, N, K)
  // bytes (16-byte aligned) for the E8M0 scale-factor images
  uint8_t* sf_images;
};
constexpr int kGemmBf16 = 16;  // internal mode id, outside fp8rl_gran

// LSE partials the GEMM leaves per token (one per column slot of each
// 256-wide vocabulary tile).
int64_t gemm_partials_per_token(int64_t N);
// Scratch the GEMM needs for the E8M0 scale-factor images of the UE8M0 mode
// (a multiple of 256 bytes).
size_t gemm_ue8m0_image_bytes(int64_t M, int64_t N, int64_t K);
cudaError_t launch_gemm_lse(const GemmArgs& a, cudaStream_t s);
cudaError_t launch_gemm_dlogits(const GemmArgs& a, cudaStream_t s);
cudaError_t launch_gemm_dense_dlogits(const GemmArgs& a, cudaStream_t s);
cudaError_t launch_gemm_store(const GemmArgs& a, cudaStream_t s);
struct BwdLayout {
  int64_t vp, tp;  // V and T rounded up to multiples of 128 (the K extents)
  // byte offsets in the workspace: codes and scales of P [T][vp], P^T [V][tp],
  // W^T [H][vp], h^T [H][tp]; E8M0 scale images of the UE8M0 recompute
  size_t p, ps, pt, pts, wt, wts, ht, hts, sf, total;
};
BwdLayout bwd_layout(int64_t T, int64_t H, int64_t V);
cudaError_t launch_lm_head_backward(const uint8_t* hc, const float* hs, const uint8_t* wc,
                                    const float* wsc, int gran, int64_t T, int64_t H, int64_t V,
                                    const int32_t* targets, const float* lse, const float* grad,
                                    const uint16_t* h, const uint16_t* W, float* dh, float* dW,
                                    bool accumulate_dw, bool pow2_scales, void* ws, cudaStream_t s);
// codes [cols][ld_out] of the transposed bf16 matrix in [rows][ld_in] with
// 128 x 128 E4M3 blocks, scales [ceil(cols/128)][ld_out/128]; columns
// rows .. ld_out-1 of the codes are zero (ld_out a multiple of 128, >= rows);
// pow2: power-of-two scales floored at 2^-127
cudaError_t launch_transpose_quantize(const uint16_t* in, int64_t rows, int64_t cols, int64_t ld_in,
                                      uint8_t* codes, float* scales, int64_t ld_out, bool pow2,
                                      cudaStream_t s);
uint32_t backward_status_take();
cudaError_t launch_combine(const float2* partials, const float* zy, const int32_t* targets,
                           const float* logp_old, float* logp, float* lse, float* ratio,
                           int64_t M, int64_t N, cudaStream_t s);
cudaError_t launch_ratios(const float* lp_new, const float* lp_old, int64_t T, float* r,
                          cudaStream_t s);
cudaError_t launch_gather_rows(const uint8_t* h_codes, const float* h_scales, int gran,
                               int64_t T, int64_t H, const int32_t* targets, const float* lse,
                               const float* grad, const int64_t* rows, int64_t n_rows,
                               uint8_t* g_codes, float* g_scales, int32_t* g_targets,
                               float* g_lse, float* g_grad, cudaStream_t s);
cudaError_t launch_wait_selftest(uint64_t limit_ns, cudaStream_t s);
uint32_t gemm_status_take();
uint32_t combine_status_take();

// ---------------------------------------------------------------- calib.cu
size_t calib_workspace_bytes(int64_t T);
cudaError_t launch_calibrate(const float* r_fp8, const float* r_bf16, const float* adv,
                             const uint8_t* mask, const float* coef, int64_t T, float eps_low,
                             float eps_high, const fp8rl_calib_opts& opts,
                             fp8rl_calib_result* result, void* ws, cudaStream_t s);
uint32_t calib_status_take();

// ----------------------------------------------------------------- loss.cu
size_t surrogate_workspace_bytes(int64_t T);
// n_valid: device count of the mask's valid tokens, or NULL to count them
cudaError_t launch_surrogate(const float* r, const float* adv, const uint8_t* mask,
                             const float* w, int64_t T, float lo, float hi, const float* bounds,
                             const int64_t* n_valid, float* grad, uint8_t* clip_mask,
                             fp8rl_clip_stats* stats, void* ws, cudaStream_t s);
size_t seq_level_workspace_bytes(int64_t T, int64_t n_seq);
cudaError_t launch_seq_level(const float* logp, const float* logp_old, const float* adv_seq,
                             const uint8_t* mask, const int32_t* sid, int64_t n_seq, int64_t T,
                             float lo, float hi, const float* bounds, float* seq_ratio,
                             uint8_t* seq_clip, float* grad, fp8rl_clip_stats* stats, void* ws,
                             cudaStream_t s);
size_t seq_surrogate_workspace_bytes(int64_t T, int64_t n_seq);
cudaError_t launch_seq_surrogate(const float* r, const float* adv, const uint8_t* mask,
                                 const float* w, const int32_t* sid, int64_t n_seq, int64_t T,
                                 float lo, float hi, const float* bounds, float* grad,
                                 uint8_t* clip_mask, fp8rl_clip_stats* stats, void* ws,
                                 cudaStream_t s);
uint32_t loss_status_take();

// ----------------------------------------------------------------- diag.cu
size_t diag_workspace_bytes(int64_t T);
cudaError_t launch_clip_diag(const float* lp8, const float* lpb, const float* r8, const float* rb,
                             const float* adv, const uint8_t* mask, int64_t T, float c_lo,
                             float c_hi, fp8rl_clip_diag* out, void* ws, cudaStream_t s);
cudaError_t launch_tis(const float* lp_old, const float* lp_samp, int64_t T, float C, float* w,
                       cudaStream_t s);

// SM count of the current device (cached per device).
int sm_count();
// CTAs of `threads` threads of `kernel` that one SM holds at once (cached per
// device and kernel; at least 1): grids of kernels that give every CTA the
// same share of the work are sized to one full wave with it.
int resident_ctas(const void* kernel, int threads);

// Records `e` as the text fp8rl_last_cuda_error() returns on this thread.
void record_cuda_error(cudaError_t e);

// The driver's cuTensorMapEncodeTiled (PFN_cuTensorMapEncodeTiled_v12000), or
// null when the driver does not provide it.
void* tensormap_encoder();

}  // namespace fp8rl
