// a4: combine the GEMM's per-chunk logsumexp partials into
//   lse_t = logsumexp_v z[t][v],  logp_t = z[t][y_t] - lse_t   (§2.1)
// and, with logp_old, the importance ratio r_t = exp(logp_t - logp_old_t).
//
// partials[c][t] = (m, s): the largest logit of vocabulary chunk c for token
// t and the sum of exp(z - m) over the chunk.  A CTA takes 32 tokens; its
// eight warps split the chunks (warp w takes c = w, w + 8, ...), each lane
// merging its token's partials with the online rule
//   (m, s) + (m', s') = (max, s exp(m - max) + s' exp(m' - max)),
// and the eight results merge through shared memory in a fixed order.
#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kTok = 32;
constexpr int kWarps = 8;

__device__ __forceinline__ void merge(float& m, float& s, float2 q) {
  if (q.x > m) {
    s = s * exp2f((m - q.x) * kLog2e) + q.y;
    m = q.x;
  } else {
    s += q.y * exp2f((q.x - m) * kLog2e);
  }
}

__global__ void __launch_bounds__(kTok * kWarps) combine_kernel(
    const float2* __restrict__ partials, const float* __restrict__ zy,
    const int32_t* __restrict__ targets, const float* __restrict__ logp_old,
    float* __restrict__ logp, float* __restrict__ lse_out, float* __restrict__ ratio, int64_t M,
    int64_t N, int64_t n_chunks) {
  __shared__ float sh_m[kWarps][kTok], sh_s[kWarps][kTok];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t t = blockIdx.x * static_cast<int64_t>(kTok) + lane;
  float m = -INFINITY, s = 0.f;
  if (t < M) {
    // sixteen loads in flight per lane: the grid has only T / 32 CTAs, so
    // the bytes in flight come from depth per thread rather than from occupancy
    constexpr int kDepth = 16;
    int64_t c = w;
    for (; c + (kDepth - 1) * kWarps < n_chunks; c += kDepth * kWarps) {
      float2 q[kDepth];
#pragma unroll
      for (int u = 0; u < kDepth; ++u) q[u] = __ldg(partials + (c + u * kWarps) * M + t);
#pragma unroll
      for (int u = 0; u < kDepth; ++u) merge(m, s, q[u]);
    }
    for (; c < n_chunks; c += kWarps) merge(m, s, __ldg(partials + c * M + t));
  }
  sh_m[w][lane] = m;
  sh_s[w][lane] = s;
  __syncthreads();
  if (w != 0 || t >= M) return;
  float mx = sh_m[0][lane];
#pragma unroll
  for (int k = 1; k < kWarps; ++k) mx = fmaxf(mx, sh_m[k][lane]);
  float sum = 0.f;
#pragma unroll
  for (int k = 0; k < kWarps; ++k) {
    const float sk = sh_s[k][lane];
    if (sk > 0.f) sum += sk * exp2f((sh_m[k][lane] - mx) * kLog2e);
  }
  const float l = mx + logf(sum);
  const int32_t y = targets[t];
  float lp;
  if (y >= 0 && y < N) {
    lp = zy[t] - l;
  } else {
    lp = NAN;
    atomicOr(&d_status, kErrDevice);
  }
  logp[t] = lp;
  if (lse_out) lse_out[t] = l;
  if (ratio) ratio[t] = expf(lp - logp_old[t]);
}

}  // namespace

cudaError_t launch_combine(const float2* partials, const float* zy, const int32_t* targets,
                           const float* logp_old, float* logp, float* lse, float* ratio,
                           int64_t M, int64_t N, cudaStream_t s) {
  if (M == 0) return cudaSuccess;
  const int64_t n_chunks = gemm_partials_per_token(N);
  const unsigned grid = static_cast<unsigned>((M + kTok - 1) / kTok);
  combine_kernel<<<grid, kTok * kWarps, 0, s>>>(partials, zy, targets, logp_old, logp, lse, ratio,
                                                M, N, n_chunks);
  return cudaGetLastError();
}

uint32_t combine_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
