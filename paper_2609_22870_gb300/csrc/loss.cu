// a6/a7: clipped surrogate with TIS weights (Eq. 1, Eq. 4), token-mean
// aggregation, clip counts by advantage sign and dloss/dlogp.
//
//   l_t = -w_t min(r_t A_t, clip(r_t, L, H) A_t)        (float64)
//   loss = sum_valid l_t / n_valid
//   clipped (gradient zeroed, §2.1): A > 0 and r >= H, or A < 0 and r <= L
//   g_t = dloss/dlogp_t = -w_t A_t r_t / n_valid on unclipped valid tokens
//
// Two grid-stride passes: the valid-token count (g needs it), then the fused
// per-token pass writing g and the clip mask.  Block partials are reduced in
// a fixed order by the last block, so the float64 loss is bit-reproducible for
// a given T.
#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr int kThreads = 256;

struct Partial {
  double loss;
  unsigned long long n_pos, n_neg, c_pos, c_neg;
  unsigned long long pad[3];
};

struct Work {
  unsigned long long n_valid;
  unsigned int ticket;
  unsigned int pad;
  Partial part[1];  // [grid]
};

int grid_of(int64_t T) {
  int64_t want = (T + kThreads * 4 - 1) / (kThreads * 4);
  const int64_t cap = static_cast<int64_t>(sm_count()) * 4;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

__global__ void __launch_bounds__(kThreads) count_valid_kernel(const uint8_t* __restrict__ mask,
                                                               int64_t T, Work* w) {
  unsigned long long n = 0;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x)
    n += mask ? (mask[t] != 0) : 1;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if ((threadIdx.x & 31) == 0 && n) atomicAdd(&w->n_valid, n);
}

template <typename T>
__device__ __forceinline__ T block_sum(T v, T* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) sh[wid] = v;
  __syncthreads();
  T r = 0;
  if (threadIdx.x == 0)
    for (int i = 0; i < kThreads / 32; ++i) r += sh[i];  // fixed order
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kThreads) surrogate_kernel(
    const float* __restrict__ r, const float* __restrict__ adv, const uint8_t* __restrict__ mask,
    const float* __restrict__ wts, int64_t T, float lo_arg, float hi_arg,
    const float* __restrict__ bounds, float* __restrict__ grad, uint8_t* __restrict__ clip_mask,
    fp8rl_clip_stats* __restrict__ stats, Work* w) {
  __shared__ double sh_d[kThreads / 32];
  __shared__ unsigned long long sh_u[kThreads / 32];
  __shared__ bool last;
  const float lo = bounds ? bounds[0] : lo_arg;
  const float hi = bounds ? bounds[1] : hi_arg;
  const unsigned long long n_valid = w->n_valid;
  const float inv_n = n_valid ? 1.0f / static_cast<float>(n_valid) : 0.f;
  double loss = 0.0;
  unsigned long long n_pos = 0, n_neg = 0, c_pos = 0, c_neg = 0;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x) {
    const bool valid = mask ? mask[t] != 0 : true;
    const float rt = r[t], at = adv[t];
    const float wt = wts ? wts[t] : 1.f;
    const bool up = valid && at > 0.f && rt >= hi;
    const bool dn = valid && at < 0.f && rt <= lo;
    float g = 0.f;
    if (valid) {
      const double rd = rt, ad = at;
      const double cl = fmin(fmax(rd, static_cast<double>(lo)), static_cast<double>(hi));
      loss += -static_cast<double>(wt) * fmin(rd * ad, cl * ad);
      n_pos += at > 0.f;
      n_neg += at < 0.f;
      c_pos += up;
      c_neg += dn;
      if (!(up || dn)) g = -(wt * at) * rt * inv_n;
    }
    if (grad) grad[t] = g;
    if (clip_mask) clip_mask[t] = static_cast<uint8_t>((up ? FP8RL_CLIP_HI : 0) | (dn ? FP8RL_CLIP_LO : 0));
  }
  loss = block_sum(loss, sh_d);
  n_pos = block_sum(n_pos, sh_u);
  n_neg = block_sum(n_neg, sh_u);
  c_pos = block_sum(c_pos, sh_u);
  c_neg = block_sum(c_neg, sh_u);
  if (threadIdx.x == 0) {
    Partial& p = w->part[blockIdx.x];
    p.loss = loss;
    p.n_pos = n_pos;
    p.n_neg = n_neg;
    p.c_pos = c_pos;
    p.c_neg = c_neg;
    __threadfence();
    last = atomicAdd(&w->ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (last && threadIdx.x == 0) {
    __threadfence();
    double L = 0.0;
    unsigned long long np = 0, nn = 0, cp = 0, cn = 0;
    for (unsigned b = 0; b < gridDim.x; ++b) {  // fixed order
      const volatile Partial& p = w->part[b];
      L += p.loss;
      np += p.n_pos;
      nn += p.n_neg;
      cp += p.c_pos;
      cn += p.c_neg;
    }
    fp8rl_clip_stats s;
    s.loss_sum = L;
    s.loss = n_valid ? L / static_cast<double>(n_valid) : 0.0;
    s.n_valid = static_cast<int64_t>(n_valid);
    s.n_pos = static_cast<int64_t>(np);
    s.n_neg = static_cast<int64_t>(nn);
    s.clipped_pos = static_cast<int64_t>(cp);
    s.clipped_neg = static_cast<int64_t>(cn);
    s.lo = lo;
    s.hi = hi;
    s.flags = n_valid ? 0 : 1;
    s.reserved = 0;
    *stats = s;
  }
}

}  // namespace

size_t surrogate_workspace_bytes(int64_t T) {
  return align_up(sizeof(Work) + sizeof(Partial) * static_cast<size_t>(grid_of(T)), 256);
}

cudaError_t launch_surrogate(const float* r, const float* adv, const uint8_t* mask,
                             const float* w, int64_t T, float lo, float hi, const float* bounds,
                             float* grad, uint8_t* clip_mask, fp8rl_clip_stats* stats, void* ws,
                             cudaStream_t s) {
  Work* work = static_cast<Work*>(ws);
  cudaError_t e = cudaMemsetAsync(work, 0, sizeof(Work), s);
  if (e != cudaSuccess) return e;
  const int grid = grid_of(T);
  count_valid_kernel<<<grid, kThreads, 0, s>>>(mask, T, work);
  surrogate_kernel<<<grid, kThreads, 0, s>>>(r, adv, mask, w, T, lo, hi, bounds, grad, clip_mask,
                                              stats, work);
  return cudaGetLastError();
}

uint32_t loss_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
