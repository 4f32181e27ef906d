/*
 * fp8rl.h -- C ABI of libfp8rl.so: FP8 token scoring followed by Calibrated
 * Clipping, as in "Towards Full Pipeline FP8 Reinforcement Learning for LLMs".
 *
 * The library runs every step on the GPU (NVIDIA GB300, sm_103a).  All tensor
 * pointers are DEVICE pointers owned by the caller unless a comment says
 * "host".  The library keeps no device allocation of its own besides a few
 * status words and the fixed scratch array of fp8rl_token_logprobs_noalloc;
 * scratch memory comes from the caller as a workspace whose size the matching
 * *_workspace_size() query returns (any alignment of 256 bytes or more; the
 * library zeroes what it needs itself).
 *
 * Every compute call is asynchronous on `stream` (a cudaStream_t; NULL is the
 * legacy default stream) and returns host-detectable errors synchronously:
 * null pointers, unsupported shapes, misalignment, a short workspace, a
 * failed launch.  Errors found by a kernel (bad target ids, non-finite or
 * negative inputs where the method forbids them, an expired bounded wait) set
 * a device status word and never trap; fp8rl_check() reports and clears it.
 * Outputs of a call that flagged an error are unspecified (NaN where noted).
 * No C++ exception crosses this interface.  No compute call synchronises with
 * the host or allocates device memory, so a sequence of calls (e.g. one
 * training step) can be captured into a CUDA graph and replayed, once each
 * call has run outside the capture on the device (the first call sets kernel
 * attributes and looks up library addresses).
 *
 * Paper references are to sections, equations and Algorithm 1 of the paper.
 */
#ifndef FP8RL_H_
#define FP8RL_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum fp8rl_status {
  FP8RL_OK = 0,
  FP8RL_EINVAL = 1,     /* null pointer, unknown enum value, negative size       */
  FP8RL_ESHAPE = 2,     /* shape outside what the call supports                  */
  FP8RL_EALIGN = 3,     /* pointer or leading dimension not 16-byte aligned      */
  FP8RL_EWORKSPACE = 4, /* workspace null or smaller than the size query         */
  FP8RL_ECUDA = 5,      /* a CUDA runtime / driver call failed                   */
  FP8RL_EDEVICE = 6,    /* a kernel flagged bad input data (from fp8rl_check)    */
  FP8RL_ETIMEOUT = 7    /* a bounded in-kernel wait expired (from fp8rl_check)   */
} fp8rl_status;

/* Scaling granularity of Eq. 3 (§2.2): one scale per tensor, per row, or per
 * block.  For the lm_head operands "row" means one scale per token of h[T][H]
 * and one per vocabulary row (output channel) of W[V][H]; "block" means 1x128
 * blocks of h and 128x128 blocks of W.
 * FP8RL_GRAN_BLOCK_UE8M0 is the block layout with power-of-two scales (the
 * codes and scales of fp8rl_quantize_ue8m0 at FP8RL_GRAN_BLOCK), a variant
 * outside the paper: the scoring calls then apply the scales in the tensor
 * cores' block-scaled MMA (E8M0 scale factors) instead of promoting each
 * 128-wide K block in registers.  Accepted by the scoring calls
 * (fp8rl_token_logprobs and its halves, the no-alloc variant, dlogits rows,
 * the lm_head backward) and by fp8rl_scales_count; the quantisers take
 * FP8RL_GRAN_BLOCK. */
typedef enum fp8rl_gran {
  FP8RL_GRAN_TENSOR = 0,
  FP8RL_GRAN_ROWWISE = 1,
  FP8RL_GRAN_BLOCK = 2,
  FP8RL_GRAN_BLOCK_UE8M0 = 3
} fp8rl_gran;

/* Operand role, which fixes the block shape and scale layout in block mode. */
typedef enum fp8rl_role {
  FP8RL_ROLE_ACT = 0,    /* hidden states h[T][H]: 1x128 blocks    */
  FP8RL_ROLE_WEIGHT = 1  /* lm_head weight W[V][H]: 128x128 blocks */
} fp8rl_role;

/* ---------------------------------------------------------------------- */
/* Status                                                                   */
/* ---------------------------------------------------------------------- */

/* Synchronises `stream`, then reads and clears the device status words that
 * kernels of this library set.  Returns FP8RL_ETIMEOUT if any bounded wait
 * expired, else FP8RL_EDEVICE if any kernel flagged bad input, else
 * FP8RL_ECUDA if the synchronisation failed, else FP8RL_OK. */
fp8rl_status fp8rl_check(void* stream);

/* Static description of a status code (never NULL). */
const char* fp8rl_status_string(fp8rl_status status);

/* Text of the last CUDA error seen by the calling host thread inside this
 * library ("" if none).  Valid until the next call on the same thread. */
const char* fp8rl_last_cuda_error(void);

/* ---------------------------------------------------------------------- */
/* a1/a2: scaled E4M3 quantisation (Eq. 3, §2.2)                            */
/* ---------------------------------------------------------------------- */

/* Number of float scales fp8rl_quantize writes for this shape (0 on bad
 * arguments):
 *   TENSOR              1                       scales[0]
 *   ROWWISE             rows                    scales[r]
 *   BLOCK, ROLE_ACT     rows * (cols/128)       scales[kb * rows + r]   (block-column major)
 *   BLOCK, ROLE_WEIGHT  ceil(rows/128)*(cols/128) scales[rb * (cols/128) + kb]
 */
int64_t fp8rl_scales_count(int64_t rows, int64_t cols, fp8rl_gran gran, fp8rl_role role);

size_t fp8rl_quantize_workspace_size(int64_t rows, int64_t cols, fp8rl_gran gran, fp8rl_role role);

/* Eq. 3: S = max|X| / 448 over each block, codes = Q_FP8(X / S).
 *   x       bf16 [rows][ld] row-major (first `cols` of each row are used);
 *           16-byte aligned, ld % 8 == 0
 *   codes   E4M3 bytes [rows][cols] row-major, 16-byte aligned
 *   scales  float32, count and layout as fp8rl_scales_count() says
 * S = fl32(amax / 448) (S = 1 when amax == 0); each code is the
 * round-to-nearest-even, saturating (+-448) E4M3 encoding of the correctly
 * rounded float32 quotient x / S.  Requires cols % 16 == 0, and cols % 128 == 0
 * in block mode.  A tail block of W along rows (rows % 128 != 0) takes its
 * amax over the rows present.  Non-finite x sets FP8RL_EDEVICE. */
fp8rl_status fp8rl_quantize(const void* x, int64_t rows, int64_t cols, int64_t ld,
                            fp8rl_gran gran, fp8rl_role role,
                            uint8_t* codes, float* scales,
                            void* workspace, size_t workspace_bytes, void* stream);

/* fp8rl_quantize with power-of-two (UE8M0) scales, a variant outside the paper
 * (whose S is amax / 448): the scale format the hardware's block-scaled MMA
 * takes.  S = 2^ceil(log2(fl32(amax / 448))), the smallest power of two not
 * below the paper's scale (1 for an all-zero group), so |x / S| <= 448 and
 * x / S is exact; codes = Q_FP8(x / S).  Arguments, layouts, workspace and
 * errors are those of fp8rl_quantize; the codes and scales feed
 * fp8rl_token_logprobs at the same granularity like any other. */
fp8rl_status fp8rl_quantize_ue8m0(const void* x, int64_t rows, int64_t cols, int64_t ld,
                                  fp8rl_gran gran, fp8rl_role role,
                                  uint8_t* codes, float* scales,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------- */
/* a3/a4: FP8 lm_head scoring with online logsumexp and target gather       */
/* ---------------------------------------------------------------------- */

/* The token ratio of §2.1 needs pi(y_t | h_t) under the FP8 forward pass of §3:
 *   z[t][v]  = sum_k S_h S_W q_h[t][k] q_W[v][k]   (fp32 accumulation on the
 *              FP8 tensor cores; in block mode per 128-wide K block)
 *   lse[t]   = log sum_v exp(z[t][v])
 *   logp[t]  = z[t][y_t] - lse[t]
 *   ratio[t] = exp(logp[t] - logp_old[t])
 * computed without ever storing z: each 128-column vocabulary chunk leaves
 * one (max, sum-exp) pair per token in the workspace, merged afterwards.
 *
 *   h_codes/h_scales  from fp8rl_quantize(h[T][H], gran, FP8RL_ROLE_ACT)
 *   w_codes/w_scales  from fp8rl_quantize(W[V][H], gran, FP8RL_ROLE_WEIGHT)
 *   targets           int32 [T], each in [0, V)  (else FP8RL_EDEVICE, logp NaN)
 *   logp_old          float [T] or NULL
 *   logp              float [T] out
 *   lse               float [T] out, or NULL
 *   ratio             float [T] out, or NULL (needs logp_old)
 * Requires T >= 1, V >= 1, H >= 16, H % 16 == 0 (H % 128 == 0 in block mode),
 * code pointers 16-byte aligned.  Temperature 1.
 * With FP8RL_GRAN_BLOCK_UE8M0 the workspace also holds the E8M0 scale-factor
 * images the block-scaled MMA reads (one byte per token, or per vocabulary
 * row block, and K block, laid out for the tensor memory; about (T + V)*H/128
 * bytes), and a scale that is not a power of two in E8M0's range
 * (2^-127 .. 2^127) sets FP8RL_EDEVICE. */
size_t fp8rl_token_logprobs_workspace_size(int64_t T, int64_t H, int64_t V, fp8rl_gran gran);

fp8rl_status fp8rl_token_logprobs(const uint8_t* h_codes, const float* h_scales,
                                  const uint8_t* w_codes, const float* w_scales,
                                  fp8rl_gran gran, int64_t T, int64_t H, int64_t V,
                                  const int32_t* targets, const float* logp_old,
                                  float* logp, float* lse, float* ratio,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* The two halves of fp8rl_token_logprobs, for callers that time or overlap
 * them separately: the FP8 GEMM with its streaming logsumexp epilogue leaves
 * per-chunk partials and z[t][y_t] in the workspace; the combine merges them.
 * Pass the same arguments and workspace to both, in this order. */
fp8rl_status fp8rl_logit_partials(const uint8_t* h_codes, const float* h_scales,
                                  const uint8_t* w_codes, const float* w_scales,
                                  fp8rl_gran gran, int64_t T, int64_t H, int64_t V,
                                  const int32_t* targets,
                                  void* workspace, size_t workspace_bytes, void* stream);

fp8rl_status fp8rl_combine_logprobs(int64_t T, int64_t H, int64_t V, fp8rl_gran gran,
                                    const int32_t* targets, const float* logp_old,
                                    float* logp, float* lse, float* ratio,
                                    void* workspace, size_t workspace_bytes, void* stream);

/* fp8rl_token_logprobs without a caller workspace.  The paper has no
 * counterpart: this call exists for callers that may not allocate device
 * memory at the point where they score tokens -- serving loops and other hot
 * paths that forbid allocation there (cudaMalloc / cudaFree can synchronise
 * the whole device and stall every stream), or processes whose device memory
 * is all reserved up front by another allocator -- and so cannot provide the
 * workspace fp8rl_token_logprobs needs.  Arguments and results are those of
 * fp8rl_token_logprobs (same kernels, same bits).
 *
 * The scratch is one array of FP8RL_NOALLOC_SCRATCH_BYTES compiled into the
 * library; every GPU that loads the library holds it until the process exits.
 * Shapes whose fp8rl_token_logprobs_workspace_size() exceeds it are refused
 * with FP8RL_EWORKSPACE (about T <= 1760 tokens at V = 151936; T <= 64000 at
 * V = 4096).  The call allocates nothing.  Its first call on a device (and the
 * first after the device's context was reset) looks up the array's device
 * address with cudaGetSymbolAddress; make that first call before any stream
 * capture.  All calls share the array and it keeps the last call's contents
 * (no part of it needs to start at zero): calls that can overlap on the GPU
 * (other streams, other host threads) race on it and must be ordered by the
 * caller. */
#define FP8RL_NOALLOC_SCRATCH_BYTES (16u << 20)

fp8rl_status fp8rl_token_logprobs_noalloc(const uint8_t* h_codes, const float* h_scales,
                                          const uint8_t* w_codes, const float* w_scales,
                                          fp8rl_gran gran, int64_t T, int64_t H, int64_t V,
                                          const int32_t* targets, const float* logp_old,
                                          float* logp, float* lse, float* ratio, void* stream);

/* The BF16 shadow pass of §4 / Algorithm 1: the reference ratios r_BF16 that
 * Calibrated Clipping matches come from forward passes in BF16.  This scores
 * the sampled tokens from the unquantised operands,
 *   z[t][v] = sum_k h[t][k] W[v][k]   (BF16 x BF16 products, fp32 accumulation
 *                                       on the tensor cores)
 * with the same streaming logsumexp + target gather as fp8rl_token_logprobs
 * (z is never stored), then logp, lse and ratio exactly as there.
 *   h   bf16 [T][ld_h] row-major (first H of each row used), 16-byte aligned
 *   W   bf16 [V][ld_w] row-major (the lm_head weight), 16-byte aligned
 *   ld_h, ld_w  row strides in elements, multiples of 8, >= H
 *   targets, logp_old, logp, lse, ratio  as for fp8rl_token_logprobs
 * Requires T >= 1, V >= 1, H >= 64 and H % 64 == 0.  The workspace (sized by
 * fp8rl_bf16_token_logprobs_workspace_size) holds the per-chunk partials. */
size_t fp8rl_bf16_token_logprobs_workspace_size(int64_t T, int64_t H, int64_t V);

fp8rl_status fp8rl_bf16_token_logprobs(const void* h, int64_t ld_h, const void* W, int64_t ld_w,
                                       int64_t T, int64_t H, int64_t V,
                                       const int32_t* targets, const float* logp_old,
                                       float* logp, float* lse, float* ratio,
                                       void* workspace, size_t workspace_bytes, void* stream);

/* r_t = exp(logp_new_t - logp_old_t) (§2.1), float [T]. */
fp8rl_status fp8rl_importance_ratios(const float* logp_new, const float* logp_old,
                                     int64_t T, float* ratio, void* stream);

/* ---------------------------------------------------------------------- */
/* a5: Calibrated Clipping (§4, Eq. 5, Algorithm 1)                         */
/* ---------------------------------------------------------------------- */

typedef enum fp8rl_calib_mode {
  FP8RL_CALIB_EXACT = 0, /* search every float32 threshold in I_L / I_H (default) */
  FP8RL_CALIB_GRID = 1   /* Algorithm 1's grid with step `step`                  */
} fp8rl_calib_mode;

/* Host-side options; fp8rl_default_calib_opts() fills the paper's values. */
typedef struct fp8rl_calib_opts {
  int32_t mode;          /* fp8rl_calib_mode                                   */
  int32_t reserved;      /* must be 0                                          */
  double lo_min, lo_max; /* I_L = [0.5, 0.9]                                   */
  double hi_min, hi_max; /* I_H = [1.2, 2.0]                                   */
  double step;           /* Delta = 0.02 (grid mode)                           */
  double delta_lo;       /* SmoothUpdate limit for L, 0.05                     */
  double delta_hi;       /* SmoothUpdate limit for H, 0.1                      */
  float lo_old, hi_old;  /* previous bounds; NaN = none (new = searched bound) */
} fp8rl_calib_opts;

/* Written to device memory by fp8rl_calibrate_clip_bounds.  The first two
 * fields are the bounds to clip with, so (const float*)result can be passed as
 * `bounds` to fp8rl_clipped_surrogate. */
typedef struct fp8rl_calib_result {
  float lo_new, hi_new;   /* SmoothUpdate(L_old, L*, dL), SmoothUpdate(H_old, H*, dH) */
  float lo_star, hi_star; /* searched bounds L*, H*                                   */
  float c_lo, c_hi;       /* reference bounds fl32(1 - eps_low), fl32(1 + eps_high)   */
  int32_t flags;          /* FP8RL_CALIB_FLAG_* bits                                  */
  int32_t shift;          /* fixed-point shift s of the Eq. 5 sums                    */
  int64_t n_neg, n_pos;   /* valid tokens with A < 0, A > 0                           */
  int64_t k_bf16;         /* #{A<0 : r_bf16 <= c_lo}  (alpha_low = k_bf16 / n_neg)    */
  int64_t k_fp8;          /* #{A<0 : r_fp8 <= L*}                                     */
  int64_t sum_pos_bf16;   /* N_bf  = sum_{A>0, r_bf16 < c_hi} q   (q = RNE(e 2^s))    */
  int64_t sum_neg_bf16;   /* D_bf  = |sum_{A<0, r_bf16 > c_lo} q|                     */
  int64_t sum_neg_fp8;    /* D_fp8 = |sum_{A<0, r_fp8 > L*} q|                        */
  int64_t sum_pos_fp8;    /* P     = sum_{A>0, r_fp8 < H*} q                          */
  double rho_bf16;        /* N_bf / D_bf                                              */
  double rho_fp8;         /* P / D_fp8                                                */
  int64_t n_valid;        /* valid tokens (mask != 0; T without a mask), for the
                             surrogate's token mean (fp8rl_clipped_surrogate)         */
} fp8rl_calib_result;

#define FP8RL_CALIB_FLAG_NO_NEG 1       /* no A<0 token: L* = c_lo (clamped to I_L) */
#define FP8RL_CALIB_FLAG_NO_POS 2       /* no A>0 token: H* = c_hi (clamped to I_H) */
#define FP8RL_CALIB_FLAG_ZERO_D_BF16 4  /* D_bf = 0: rho_BF16 undefined, H* = c_hi  */
#define FP8RL_CALIB_FLAG_ZERO_D_FP8 8   /* D_fp8 = 0: rho_FP8 undefined, H* = c_hi  */

void fp8rl_default_calib_opts(fp8rl_calib_opts* opts);

/* The workspace holds the search state (33 KB) and, for EXACT mode, lists of
 * the tokens whose ratios fall inside I_L and I_H: 16 bytes per token of
 * capacity (T entries each, so any input fits). */
size_t fp8rl_calibrate_workspace_size(int64_t T);

/* Algorithm 1.  Inputs, float [T] unless noted:
 *   r_fp8, r_bf16  importance ratios from the FP8 path and the BF16 shadow pass
 *   adv            advantages A_t
 *   mask           uint8 [T], 1 = valid token (NULL = all valid)
 *   coef           w_t^TIS * pi_sampler(y_t|h_t) of Eq. 5 (NULL = 1)
 *   opts           HOST pointer, NULL = fp8rl_default_calib_opts()
 *   result         DEVICE pointer to one fp8rl_calib_result
 * Stage 1 (§4): k = #{A<0 : r_bf16 <= c_lo}; L* minimises
 * |#{A<0 : r_fp8 <= L} - k| over L in I_L (every float32 in EXACT mode, the
 * grid in GRID mode); among minimisers the one nearest c_lo, then the smaller.
 * Stage 2 (Eq. 5): e_t = (coef_t r_t) A_t in float64, rounded to integers
 * q_t = RNE(e_t 2^s) with one shift s per call so no sum overflows; H*
 * minimises |P(H) D_bf - N_bf D_fp8| (= |rho_FP8 - rho_BF16| D_bf D_fp8) over H
 * in I_H, ties to the point nearest c_hi, then the smaller.  Then SmoothUpdate.
 * Ratios and coef must be finite and >= 0, advantages finite (else
 * FP8RL_EDEVICE).  T >= 0. */
fp8rl_status fp8rl_calibrate_clip_bounds(const float* r_fp8, const float* r_bf16,
                                         const float* adv, const uint8_t* mask,
                                         const float* coef, int64_t T,
                                         float eps_low, float eps_high,
                                         const fp8rl_calib_opts* opts,
                                         fp8rl_calib_result* result,
                                         void* workspace, size_t workspace_bytes,
                                         void* stream);

/* ---------------------------------------------------------------------- */
/* a6/a7: clipped surrogate, clip fractions, dLoss/dlogp (Eq. 1, Eq. 4)      */
/* ---------------------------------------------------------------------- */

/* Device-resident statistics of one fp8rl_clipped_surrogate call. */
typedef struct fp8rl_clip_stats {
  double loss;           /* sum_valid l_t / n_valid (0 when n_valid == 0) */
  double loss_sum;       /* sum_valid l_t                                 */
  int64_t n_valid, n_pos, n_neg;
  int64_t clipped_pos;   /* A > 0 and r >= H   */
  int64_t clipped_neg;   /* A < 0 and r <= L   */
  float lo, hi;          /* bounds used        */
  int32_t flags;         /* 1 = no valid token */
  int32_t n_seq_valid;   /* sequence-mean call: sequences with a valid token (S); else 0 */
  /* Clip fractions (§3; PPO's clip fraction split by advantage sign), each 0
   * when its denominator is 0, float64 quotients of the exact counts:       */
  double clip_frac_pos;  /* clipped_pos / n_pos                              */
  double clip_frac_neg;  /* clipped_neg / n_neg                              */
  double clip_frac;      /* (clipped_pos + clipped_neg) / n_valid; for
                            sequence-level clipping / n_seq_valid (responses) */
} fp8rl_clip_stats;

#define FP8RL_CLIP_HI 1  /* clip-mask bit: A > 0 and r >= H */
#define FP8RL_CLIP_LO 2  /* clip-mask bit: A < 0 and r <= L */

size_t fp8rl_surrogate_workspace_size(int64_t T);

/* l_t = -w_t min(r_t A_t, clip(r_t, L, H) A_t) (Eq. 1 with the TIS weight of
 * Eq. 4 and calibrated bounds), loss = sum_valid l_t / n_valid (token mean;
 * float32 terms summed with compensation per thread, float64 across threads
 * in a fixed order: deterministic for a given T on a given device).
 *   r, adv       float [T];  mask uint8 [T] or NULL;  w_tis float [T] or NULL (1)
 *   lo, hi       bounds by value, used when `bounds` is NULL
 *   bounds       DEVICE float[2] {L, H} or NULL (e.g. a fp8rl_calib_result*)
 *   n_valid      DEVICE int64, the number of valid tokens of `mask` when the
 *                caller has it (e.g. &result->n_valid of fp8rl_calibrate_clip_bounds
 *                on the same mask), read at run time; NULL: the call counts
 *                them in a pass of its own.  Ignored without a mask (T).
 *   grad_logp    float [T] out or NULL: dloss/dlogp_t = -w A r / n_valid on
 *                unclipped valid tokens, 0 elsewhere.  With lse from
 *                fp8rl_token_logprobs this is dLoss/dlogits in factored form:
 *                dLoss/dz[t][v] = grad_logp[t] (1{v == y_t} - exp(z[t][v] - lse[t])).
 *   clip_mask    uint8 [T] out or NULL: FP8RL_CLIP_HI / FP8RL_CLIP_LO bits
 *   stats        DEVICE pointer to one fp8rl_clip_stats */
fp8rl_status fp8rl_clipped_surrogate(const float* r, const float* adv, const uint8_t* mask,
                                     const float* w_tis, int64_t T, float lo, float hi,
                                     const float* bounds, const int64_t* n_valid,
                                     float* grad_logp, uint8_t* clip_mask,
                                     fp8rl_clip_stats* stats,
                                     void* workspace, size_t workspace_bytes, void* stream);

/* The same surrogate with GRPO's per-response normalisation (§2.1: each
 * response's token terms are averaged, 1/|o_i| sum_t, then the responses):
 *   loss = (1/S) sum_{i : n_i > 0} (1/n_i) sum_{t in i, valid} l_t
 *   g_t  = -w_t A_t r_t / (S n_i) on unclipped valid tokens, 0 elsewhere
 * n_i = valid tokens of sequence i, S = sequences with n_i > 0 (written to
 * stats->n_seq_valid); loss_sum = S * loss.  seq_id int32 [T] gives each
 * token's sequence in [0, n_seq) (tokens of a sequence need not be
 * contiguous); an id outside that range sets FP8RL_EDEVICE and the token counts
 * nowhere.  Other arguments, outputs and the clip semantics are those of
 * fp8rl_clipped_surrogate; the workspace size depends on n_seq. */
size_t fp8rl_surrogate_seq_mean_workspace_size(int64_t T, int64_t n_seq);

fp8rl_status fp8rl_clipped_surrogate_seq_mean(const float* r, const float* adv,
                                              const uint8_t* mask, const float* w_tis,
                                              const int32_t* seq_id, int64_t n_seq, int64_t T,
                                              float lo, float hi, const float* bounds,
                                              float* grad_logp, uint8_t* clip_mask,
                                              fp8rl_clip_stats* stats,
                                              void* workspace, size_t workspace_bytes,
                                              void* stream);

/* Sequence-level ratio clipping: the response-level trust region that §6
 * (related work) names, with one ratio per response instead of per token.
 * For sequence i with n_i valid tokens:
 *   s_i  = exp((1/n_i) sum_{t in i, valid} d_t),  d_t = logp_t - logp_old_t
 *          (the geometric mean of the token ratios), rounded to float32
 *   loss = (1/S) sum_{i : n_i > 0} -A_i m_i,  m_i = min(s_i, H) if A_i >= 0, else max(s_i, L)
 *   clipped (gradient zeroed): A_i > 0 and s_i >= H, or A_i < 0 and s_i <= L
 *   g_t  = dloss/dlogp_t = -A_i s_i / (n_i S) on valid tokens of unclipped
 *          sequences (float64 quotient rounded to float32), 0 elsewhere
 * S = sequences with n_i > 0.  The exponent sums are accumulated exactly on
 * the 2^-32 grid (each |d_t| >= 2^-8 is exact there, smaller ones round to
 * it), so the result is independent of token order; exact for sequences of
 * up to 2^24 valid tokens.
 *   logp, logp_old  float [T] (the scored and the old log-probs)
 *   adv_seq     float [n_seq]: the response advantages A_i
 *   mask        uint8 [T] or NULL;  seq_id int32 [T] in [0, n_seq) (tokens of
 *               a sequence need not be contiguous)
 *   lo, hi / bounds  as for fp8rl_clipped_surrogate
 *   seq_ratio   float [n_seq] out or NULL: s_i (0 for a sequence without valid tokens)
 *   seq_clip    uint8 [n_seq] out or NULL: FP8RL_CLIP_HI / FP8RL_CLIP_LO bits
 *   grad_logp   float [T] out or NULL
 *   stats       DEVICE fp8rl_clip_stats: loss, loss_sum = S loss, n_valid
 *               (tokens), n_pos / n_neg / clipped_pos / clipped_neg counted
 *               over SEQUENCES with n_i > 0, n_seq_valid = S, flags 1 when no
 *               token is valid.
 * A valid token with |d_t| > 128 or a NaN d_t (its float32 ratio would over-
 * or underflow) and an id outside [0, n_seq) set FP8RL_EDEVICE; such a d_t
 * counts as its clamp to [-128, 128] (NaN as 0), such an id nowhere. */
size_t fp8rl_seq_level_surrogate_workspace_size(int64_t T, int64_t n_seq);

fp8rl_status fp8rl_seq_level_clipped_surrogate(const float* logp, const float* logp_old,
                                               const float* adv_seq, const uint8_t* mask,
                                               const int32_t* seq_id, int64_t n_seq, int64_t T,
                                               float lo, float hi, const float* bounds,
                                               float* seq_ratio, uint8_t* seq_clip,
                                               float* grad_logp, fp8rl_clip_stats* stats,
                                               void* workspace, size_t workspace_bytes,
                                               void* stream);

/* Dense dLoss/dlogits for selected rows (a verification and debugging path;
 * the hot path keeps the factored form above).  For i < n_rows, t = rows[i]:
 *   out[i][v] = grad_logp[t] * (1{v == y_t} - exp(z[t][v] - lse[t])),  v < V,
 * with z recomputed by the same FP8 GEMM as fp8rl_token_logprobs.
 *   rows  int64 [n_rows] DEVICE, each in [0, T)    out float [n_rows][V] */
size_t fp8rl_dlogits_workspace_size(int64_t n_rows, int64_t H, int64_t V, fp8rl_gran gran);

fp8rl_status fp8rl_dlogits_rows(const uint8_t* h_codes, const float* h_scales,
                                const uint8_t* w_codes, const float* w_scales,
                                fp8rl_gran gran, int64_t T, int64_t H, int64_t V,
                                const int32_t* targets, const float* lse,
                                const float* grad_logp, const int64_t* rows, int64_t n_rows,
                                float* out, void* workspace, size_t workspace_bytes,
                                void* stream);

/* Backward through the FP8 lm_head (the chain rule of a3/a4 past the logits;
 * the paper trains with FP8 forward and backward GEMMs, §3 and the
 * performance appendix).  With g_t = grad_logp[t] (e.g. from
 * fp8rl_clipped_surrogate) and lse from fp8rl_token_logprobs:
 *   P[t][v] = g_t (1{v == y_t} - exp(z[t][v] - lse_t)),  z recomputed by the
 *             FP8 GEMM of fp8rl_token_logprobs, P in float32 (neither the
 *             logits nor P in float32 are ever stored)
 *   dh[t][k] = sum_v P[t][v] W[v][k]        float32 [T][H]
 *   dW[v][k] = sum_t P[t][v] h[t][k]        float32 [V][H]
 * The quantisers pass the gradient straight through, and both contractions
 * run on the block-scaled FP8 tensor-core GEMM with every operand
 * E4M3-quantised (Eq. 3) along its own K axis: P with 1x128 blocks along V
 * (dh), P^T with 128 x 128 blocks (dW), and the transposed bf16 operands
 * w_bf16^T [H][V] and h_bf16^T [H][T] with 128 x 128 blocks; float32
 * accumulation.  The scales of these four operands are amax / 448 (the
 * paper's format), promoted in registers per 128-wide K block; with
 * FP8RL_BWD_POW2_SCALES (implied by FP8RL_GRAN_BLOCK_UE8M0) they are rounded
 * up to powers of two (floored at 2^-127) and both contractions run on the
 * block-scaled MMA (kind::mxf8f6f4), which applies them in hardware.  The
 * recompute of z always uses the forward's codes and scales as given.
 *   h_codes ... targets   as for fp8rl_token_logprobs (any granularity)
 *   lse, grad_logp        float [T] DEVICE
 *   h_bf16, w_bf16        bf16 [T][H], [V][H], the operands the codes came from
 *   dh, dW                float out, 16-byte aligned; either may be NULL to
 *                         skip that contraction (not both)
 *   flags                 FP8RL_BWD_* bits: ACCUMULATE_DW: dW += (several
 *                         token chunks, one dW); POW2_SCALES: as above;
 *                         other bits give FP8RL_EINVAL
 * T and V below 2^31 - 256, else FP8RL_ESHAPE; misaligned h_bf16, w_bf16, dh,
 * dW or workspace give FP8RL_EALIGN; a non-finite h_bf16 or w_bf16 sets
 * FP8RL_EDEVICE.  The workspace holds the codes and scales of the four
 * quantised operands: about (T + H) V' + (V + H) T' bytes with V', T' = V, T
 * rounded up to multiples of 128 (5.72 GB at T 16384, H 4096, V 151936);
 * callers with less memory pass token chunks whose length is a multiple of
 * 128 (so the 128 x 128 blocks of P^T and h^T are those of the whole batch;
 * granularity other than per tensor, so the chunk's codes are the batch's)
 * and accumulate dW.  Target ids are not checked again here
 * (fp8rl_token_logprobs flags them): an id outside [0, V) adds no one-hot
 * term to its row of P. */
#define FP8RL_BWD_ACCUMULATE_DW 1
#define FP8RL_BWD_POW2_SCALES 2

size_t fp8rl_lm_head_backward_workspace_size(int64_t T, int64_t H, int64_t V);

fp8rl_status fp8rl_lm_head_backward(const uint8_t* h_codes, const float* h_scales,
                                    const uint8_t* w_codes, const float* w_scales,
                                    fp8rl_gran gran, int64_t T, int64_t H, int64_t V,
                                    const int32_t* targets, const float* lse,
                                    const float* grad_logp, const void* h_bf16,
                                    const void* w_bf16, float* dh, float* dW,
                                    int flags, void* workspace, size_t workspace_bytes,
                                    void* stream);

/* ---------------------------------------------------------------------- */
/* §3 diagnostics against BF16 references; TIS weights (§2.3)               */
/* ---------------------------------------------------------------------- */

/* Device-resident result of fp8rl_clip_diagnostics (counts over valid tokens). */
typedef struct fp8rl_clip_diag {
  int64_t n_valid, n_pos, n_neg;    /* mask = 1; and A > 0, A < 0 among them      */
  int64_t clipped_lo_fp8;           /* A < 0 and r_fp8  <= c_lo                  */
  int64_t clipped_hi_fp8;           /* A > 0 and r_fp8  >= c_hi                  */
  int64_t clipped_lo_bf16;          /* A < 0 and r_bf16 <= c_lo                  */
  int64_t clipped_hi_bf16;          /* A > 0 and r_bf16 >= c_hi                  */
  int64_t over_clipped_lo;          /* A < 0, r_bf16 > c_lo and r_fp8 <= c_lo     */
  int64_t over_clipped_hi;          /* A > 0, r_bf16 < c_hi and r_fp8 >= c_hi     */
  double abs_err_prob, sum_prob_bf16;   /* sum |p_fp8 - p_bf16|, sum p_bf16, p = exp(logp) */
  double abs_err_ratio, sum_ratio_bf16; /* sum |r_fp8 - r_bf16|, sum |r_bf16|             */
  double nmae_prob, nmae_ratio;     /* the quotients of the two pairs (NaN if 0/0) */
  float c_lo, c_hi;                 /* fl32(1 - eps_low), fl32(1 + eps_high)      */
  int32_t flags;                    /* FP8RL_DIAG_FLAG_* bits                     */
  int32_t reserved;
} fp8rl_clip_diag;

#define FP8RL_DIAG_FLAG_NO_VALID 1  /* no valid token                          */
#define FP8RL_DIAG_FLAG_NO_PROB 2   /* logp_fp8 / logp_bf16 not given: no prob NMAE */

size_t fp8rl_clip_diagnostics_workspace_size(int64_t T);

/* The diagnosis of §3 ("The Cause"): how often FP8 noise pushes tokens over
 * the trust-region bounds that their BF16 references stay inside
 * (over-clipping, lower: A < 0, r_BF16 > 1 - eps, r_FP8 <= 1 - eps; upper:
 * A > 0, r_BF16 < 1 + eps, r_FP8 >= 1 + eps), the PPO clip counts of both
 * ratio sets at the same bounds (clipped at equality, §2.1), and the
 * normalised mean absolute error sum |x - x_ref| / sum |x_ref| of the
 * probabilities exp(logp) and of the ratios.  One pass; counts exact, sums
 * compensated float32 per thread and float64 across threads in a fixed
 * order.
 *   logp_fp8, logp_bf16  float [T] or both NULL (no probability NMAE)
 *   r_fp8, r_bf16, adv   float [T];  mask uint8 [T] or NULL (all valid)
 *   out                  DEVICE pointer to one fp8rl_clip_diag */
fp8rl_status fp8rl_clip_diagnostics(const float* logp_fp8, const float* logp_bf16,
                                    const float* r_fp8, const float* r_bf16, const float* adv,
                                    const uint8_t* mask, int64_t T, float eps_low,
                                    float eps_high, fp8rl_clip_diag* out,
                                    void* workspace, size_t workspace_bytes, void* stream);

/* The truncated importance-sampling weight of J_TIS (§2.3), which corrects
 * for the sampler (FP8 rollout) differing from the learner's old policy:
 *   w_t = min(exp(logp_old_t - logp_sampler_t), C)       (C = 2 typically)
 * float [T] in, float [T] out (feeds fp8rl_clipped_surrogate's w_tis).
 * C must be finite and > 0. */
fp8rl_status fp8rl_tis_weights(const float* logp_old, const float* logp_sampler, int64_t T,
                               float C, float* w_tis, void* stream);

/* ---------------------------------------------------------------------- */
/* Bounded waits                                                            */
/* ---------------------------------------------------------------------- */

/* Every spin-wait in this library's kernels gives up after this many
 * nanoseconds of GPU time (default 2e9), sets FP8RL_ETIMEOUT and returns after
 * draining its own in-flight copies.  Process-wide; 0 restores the default. */
void fp8rl_set_wait_limit_ns(uint64_t limit_ns);

/* Launches one CTA that waits, with the bounded wait every kernel here uses,
 * on a barrier nothing will signal; the wait expires after `limit_ns`, so a
 * following fp8rl_check() returns FP8RL_ETIMEOUT and the context stays
 * usable.  Used to test the timeout path without hanging a GPU. */
fp8rl_status fp8rl_wait_selftest(uint64_t limit_ns, void* stream);

#ifdef __cplusplus
} /* extern "C" */
#endif

#endif /* FP8RL_H_ */
