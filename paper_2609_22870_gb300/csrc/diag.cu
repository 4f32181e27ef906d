// §3 diagnostics of full-pipeline FP8 against BF16 references, and the
// truncated importance-sampling weight of J_TIS (§2.3).
//
// clip_diag_kernel, one grid-stride pass over valid tokens (four per thread
// and step, 16-byte loads when the arrays allow):
//   over-clipping  lower: A < 0, r_bf16 > c_lo, r_fp8 <= c_lo
//                  upper: A > 0, r_bf16 < c_hi, r_fp8 >= c_hi
//   clip counts    of r_fp8 and of r_bf16 at the same bounds (at equality)
//   NMAE           sum |x - x_ref| / sum |x_ref| for the ratios and for the
//                  probabilities p = exp(logp); |p_fp8 - p_bf16| is formed as
//                  p_bf16 |expm1(logp_fp8 - logp_bf16)|, whose argument is an
//                  exact float32 difference, so no cancellation is lost.
// Counts are exact; sums are compensated float32 per thread and float64
// across threads in a fixed order by the last block (bit-reproducible for a
// given T and launch).
//
// tis_kernel: w_t = min(exp(logp_old_t - logp_sampler_t), C).
#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

constexpr int kThreads = 256;
constexpr int kCtasPerSm = 8;
constexpr int kCounts = 9;  // n_valid n_pos n_neg clo8 chi8 clob chib olo ohi
constexpr int kSums = 4;    // abs_err_prob sum_prob_bf16 abs_err_ratio sum_ratio_bf16

struct Partial {
  double sum[kSums];
  unsigned long long cnt[kCounts];
  unsigned long long pad[3];
};

struct Work {
  unsigned int ticket;
  unsigned int pad[63];
  Partial part[1];  // [grid]
};

int grid_of(int64_t T) {
  const int64_t want = (T + kThreads * 16 - 1) / (kThreads * 16);
  const int64_t cap = static_cast<int64_t>(sm_count()) * kCtasPerSm;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

// Knuth's two-sum compensated float32 accumulator: value s + c.
struct Comp {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float t = s + x;
    const float z = t - s;
    c += (s - (t - z)) + (x - z);
    s = t;
  }
};

struct Acc {
  uint32_t cnt[kCounts] = {0, 0, 0, 0, 0, 0, 0, 0, 0};
  Comp sum[kSums];
};

struct Bounds {
  float lo, hi;
};

__device__ __forceinline__ void token(float l8, float lb, float r8, float rb, float A, bool valid,
                                      bool with_p, const Bounds& b, Acc& a) {
  if (!valid) return;
  const bool neg = A < 0.f, pos = A > 0.f;
  a.cnt[0] += 1;
  a.cnt[1] += pos;
  a.cnt[2] += neg;
  a.cnt[3] += neg && r8 <= b.lo;
  a.cnt[4] += pos && r8 >= b.hi;
  a.cnt[5] += neg && rb <= b.lo;
  a.cnt[6] += pos && rb >= b.hi;
  a.cnt[7] += neg && rb > b.lo && r8 <= b.lo;
  a.cnt[8] += pos && rb < b.hi && r8 >= b.hi;
  a.sum[2].add(fabsf(r8 - rb));
  a.sum[3].add(fabsf(rb));
  if (with_p) {
    const float pb = expf(lb);
    a.sum[0].add(pb * fabsf(expm1f(l8 - lb)));
    a.sum[1].add(pb);
  }
}

template <typename V>
__device__ __forceinline__ V block_sum(V v, V* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) sh[wid] = v;
  __syncthreads();
  V r = 0;
  if (threadIdx.x == 0)
    for (int i = 0; i < kThreads / 32; ++i) r += sh[i];
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kThreads) clip_diag_kernel(
    const float* __restrict__ lp8, const float* __restrict__ lpb, const float* __restrict__ r8,
    const float* __restrict__ rb, const float* __restrict__ adv, const uint8_t* __restrict__ mask,
    int64_t T, Bounds b, fp8rl_clip_diag* __restrict__ out, Work* w, bool vec) {
  __shared__ double sh_d[kThreads / 32];
  __shared__ unsigned long long sh_u[kThreads / 32];
  __shared__ bool last;
  const bool with_p = lp8 != nullptr && lpb != nullptr;
  Acc a;
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t T4 = vec ? T / 4 : 0;
  for (int64_t i = tid; i < T4; i += stride) {
    const float4 f8 = __ldg(reinterpret_cast<const float4*>(r8) + i);
    const float4 fb = __ldg(reinterpret_cast<const float4*>(rb) + i);
    const float4 fa = __ldg(reinterpret_cast<const float4*>(adv) + i);
    const uint32_t mv = mask ? __ldg(reinterpret_cast<const uint32_t*>(mask) + i) : 0x01010101u;
    float4 l8 = make_float4(0.f, 0.f, 0.f, 0.f), lb = l8;
    if (with_p) {
      l8 = __ldg(reinterpret_cast<const float4*>(lp8) + i);
      lb = __ldg(reinterpret_cast<const float4*>(lpb) + i);
    }
    token(l8.x, lb.x, f8.x, fb.x, fa.x, (mv & 0xFFu) != 0, with_p, b, a);
    token(l8.y, lb.y, f8.y, fb.y, fa.y, (mv & 0xFF00u) != 0, with_p, b, a);
    token(l8.z, lb.z, f8.z, fb.z, fa.z, (mv & 0xFF0000u) != 0, with_p, b, a);
    token(l8.w, lb.w, f8.w, fb.w, fa.w, (mv & 0xFF000000u) != 0, with_p, b, a);
  }
  for (int64_t t = T4 * 4 + tid; t < T; t += stride)
    token(with_p ? lp8[t] : 0.f, with_p ? lpb[t] : 0.f, r8[t], rb[t], adv[t],
          mask ? mask[t] != 0 : true, with_p, b, a);
  double sums[kSums];
  unsigned long long cnts[kCounts];
#pragma unroll
  for (int k = 0; k < kSums; ++k)
    sums[k] = block_sum(static_cast<double>(a.sum[k].s) + static_cast<double>(a.sum[k].c), sh_d);
#pragma unroll
  for (int k = 0; k < kCounts; ++k) cnts[k] = block_sum<unsigned long long>(a.cnt[k], sh_u);
  if (threadIdx.x == 0) {
    Partial& p = w->part[blockIdx.x];
    for (int k = 0; k < kSums; ++k) p.sum[k] = sums[k];
    for (int k = 0; k < kCounts; ++k) p.cnt[k] = cnts[k];
    __threadfence();
    last = atomicAdd(&w->ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  // the last block reduces the partials in a fixed order
  __threadfence();
  double S[kSums] = {0.0, 0.0, 0.0, 0.0};
  unsigned long long C[kCounts] = {0, 0, 0, 0, 0, 0, 0, 0, 0};
  for (unsigned k = threadIdx.x; k < gridDim.x; k += kThreads) {
    const volatile Partial& p = w->part[k];
    for (int j = 0; j < kSums; ++j) S[j] += p.sum[j];
    for (int j = 0; j < kCounts; ++j) C[j] += p.cnt[j];
  }
#pragma unroll
  for (int j = 0; j < kSums; ++j) S[j] = block_sum(S[j], sh_d);
#pragma unroll
  for (int j = 0; j < kCounts; ++j) C[j] = block_sum(C[j], sh_u);
  if (threadIdx.x == 0) {
    fp8rl_clip_diag d;
    d.n_valid = static_cast<int64_t>(C[0]);
    d.n_pos = static_cast<int64_t>(C[1]);
    d.n_neg = static_cast<int64_t>(C[2]);
    d.clipped_lo_fp8 = static_cast<int64_t>(C[3]);
    d.clipped_hi_fp8 = static_cast<int64_t>(C[4]);
    d.clipped_lo_bf16 = static_cast<int64_t>(C[5]);
    d.clipped_hi_bf16 = static_cast<int64_t>(C[6]);
    d.over_clipped_lo = static_cast<int64_t>(C[7]);
    d.over_clipped_hi = static_cast<int64_t>(C[8]);
    d.abs_err_prob = S[0];
    d.sum_prob_bf16 = S[1];
    d.abs_err_ratio = S[2];
    d.sum_ratio_bf16 = S[3];
    d.nmae_prob = (with_p && S[1] > 0.0) ? S[0] / S[1] : NAN;
    d.nmae_ratio = S[3] > 0.0 ? S[2] / S[3] : NAN;
    d.c_lo = b.lo;
    d.c_hi = b.hi;
    d.flags = (C[0] == 0 ? FP8RL_DIAG_FLAG_NO_VALID : 0) | (with_p ? 0 : FP8RL_DIAG_FLAG_NO_PROB);
    d.reserved = 0;
    *out = d;
  }
}

__global__ void tis_kernel(const float* __restrict__ lp_old, const float* __restrict__ lp_samp,
                           int64_t T, float C, float* __restrict__ w) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x)
    w[t] = fminf(expf(lp_old[t] - lp_samp[t]), C);
}

bool aligned(const void* p, uintptr_t n) { return (reinterpret_cast<uintptr_t>(p) & (n - 1)) == 0; }

}  // namespace

size_t diag_workspace_bytes(int64_t T) {
  return align_up(sizeof(Work) + sizeof(Partial) * static_cast<size_t>(grid_of(T)), 256);
}

cudaError_t launch_clip_diag(const float* lp8, const float* lpb, const float* r8, const float* rb,
                             const float* adv, const uint8_t* mask, int64_t T, float c_lo,
                             float c_hi, fp8rl_clip_diag* out, void* ws, cudaStream_t s) {
  Work* work = static_cast<Work*>(ws);
  cudaError_t e = cudaMemsetAsync(work, 0, sizeof(unsigned int), s);
  if (e != cudaSuccess) return e;
  const bool vec = aligned(r8, 16) && aligned(rb, 16) && aligned(adv, 16) && aligned(lp8, 16) &&
                   aligned(lpb, 16) && aligned(mask, 4);
  clip_diag_kernel<<<grid_of(T), kThreads, 0, s>>>(lp8, lpb, r8, rb, adv, mask, T, Bounds{c_lo, c_hi},
                                                    out, work, vec);
  return cudaGetLastError();
}

cudaError_t launch_tis(const float* lp_old, const float* lp_samp, int64_t T, float C, float* w,
                       cudaStream_t s) {
  if (T == 0) return cudaSuccess;
  int64_t b = (T + 255) / 256;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  tis_kernel<<<static_cast<int>(b > cap ? cap : b), 256, 0, s>>>(lp_old, lp_samp, T, C, w);
  return cudaGetLastError();
}


}  // namespace fp8rl
