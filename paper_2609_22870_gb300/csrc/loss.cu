// a6/a7: clipped surrogate with TIS weights (Eq. 1, Eq. 4), token-mean
// aggregation, clip counts by advantage sign and dloss/dlogp.
//
//   l_t = -w_t min(r_t A_t, clip(r_t, L, H) A_t) = -w_t A_t m_t,
//         m_t = min(r_t, H) when A_t >= 0, max(r_t, L) when A_t < 0
//   loss = sum_valid l_t / n_valid
//   clipped (gradient zeroed, §2.1): A > 0 and r >= H, or A < 0 and r <= L
//   g_t = dloss/dlogp_t = -w_t A_t r_t / n_valid on unclipped valid tokens
//
// Two grid-stride passes: the valid-token count (g needs it; skipped without
// a mask), then the fused per-token pass writing g and the clip mask, four
// tokens per thread and step with 16-byte loads when the arrays allow.  Terms
// are float32 (two roundings of the exact product); each thread sums its
// terms with an error-free two-sum compensation (Knuth), so its partial is
// the float32 sum to within one rounding; partials meet in float64 through a
// fixed-order reduction by the last block, so the loss is bit-reproducible for
// a given T and launch.
//
// Sequence-mean variant (GRPO's per-response normalisation, §2.1): a count
// pass gives each sequence's valid tokens n_i (atomics aggregated over a warp's
// tokens of the same sequence) and S = #{i : n_i > 0}; the
// fused pass then weights each term by 1/n_i and each gradient by 1/(S n_i):
//   loss = (1/S) sum_i (1/n_i) sum_{t in i} l_t,   g_t = -w_t A_t r_t / (S n_i).
#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr int kThreads = 256;
constexpr int kCtasPerSm = 8;

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
  const int64_t want = (T + kThreads * 16 - 1) / (kThreads * 16);
  const int64_t cap = static_cast<int64_t>(sm_count()) * kCtasPerSm;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

// Number of non-zero bytes of a word.
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t w) {
  return __popc((((w & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | w) & 0x80808080u);
}

__global__ void __launch_bounds__(kThreads) count_valid_kernel(const uint8_t* __restrict__ mask,
                                                               int64_t T, Work* w) {
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  uint32_t n = 0;
  const bool vec = (reinterpret_cast<uintptr_t>(mask) & 15) == 0;
  const int64_t T16 = vec ? T / 16 : 0;
  for (int64_t i = tid; i < T16; i += stride) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(mask) + i);
    n += nonzero_bytes(v.x) + nonzero_bytes(v.y) + nonzero_bytes(v.z) + nonzero_bytes(v.w);
  }
  for (int64_t t = T16 * 16 + tid; t < T; t += stride) n += mask[t] != 0;
  const uint32_t s = __reduce_add_sync(0xffffffffu, n);
  if ((threadIdx.x & 31) == 0 && s) atomicAdd(&w->n_valid, static_cast<unsigned long long>(s));
}

// Fixed-order sum over the block; thread 0 gets the result.
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

struct Acc {
  float s = 0.f, c = 0.f;  // compensated float32 sum: value s + c
  uint32_t n_pos = 0, n_neg = 0, c_pos = 0, c_neg = 0;
  // Knuth's two-sum: s + x = t + e exactly.
  __device__ __forceinline__ void add(float x) {
    const float t = s + x;
    const float z = t - s;
    c += (s - (t - z)) + (x - z);
    s = t;
  }
};

struct Bounds {
  float lo, hi, inv_n;
};

// One token: its term, its gradient and clip-mask byte; counts into `a`.
__device__ __forceinline__ float token(float rt, float at, bool valid, float wt, const Bounds& b,
                                       Acc& a, float& g, uint32_t& cm) {
  const bool up = valid && at > 0.f && rt >= b.hi;
  const bool dn = valid && at < 0.f && rt <= b.lo;
  const float m = at >= 0.f ? fminf(rt, b.hi) : fmaxf(rt, b.lo);
  a.n_pos += valid && at > 0.f;
  a.n_neg += valid && at < 0.f;
  a.c_pos += up;
  a.c_neg += dn;
  g = (valid && !(up || dn)) ? -(wt * at) * rt * b.inv_n : 0.f;
  cm = (up ? FP8RL_CLIP_HI : 0u) | (dn ? FP8RL_CLIP_LO : 0u);
  return valid ? -(wt * (at * m)) : 0.f;
}

__global__ void __launch_bounds__(kThreads) surrogate_kernel(
    const float* __restrict__ r, const float* __restrict__ adv, const uint8_t* __restrict__ mask,
    const float* __restrict__ wts, int64_t T, float lo_arg, float hi_arg,
    const float* __restrict__ bounds, float* __restrict__ grad, uint8_t* __restrict__ clip_mask,
    fp8rl_clip_stats* __restrict__ stats, Work* w, bool vec) {
  __shared__ double sh_d[kThreads / 32];
  __shared__ unsigned long long sh_u[kThreads / 32];
  __shared__ bool last;
  Bounds b;
  b.lo = bounds ? bounds[0] : lo_arg;
  b.hi = bounds ? bounds[1] : hi_arg;
  const unsigned long long n_valid = mask ? w->n_valid : static_cast<unsigned long long>(T);
  b.inv_n = n_valid ? 1.0f / static_cast<float>(n_valid) : 0.f;
  Acc a;
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t T4 = vec ? T / 4 : 0;
  for (int64_t i = tid; i < T4; i += stride) {
    const float4 rv = __ldg(reinterpret_cast<const float4*>(r) + i);
    const float4 av = __ldg(reinterpret_cast<const float4*>(adv) + i);
    const float4 wv = wts ? __ldg(reinterpret_cast<const float4*>(wts) + i) : make_float4(1.f, 1.f, 1.f, 1.f);
    const uint32_t mv = mask ? __ldg(reinterpret_cast<const uint32_t*>(mask) + i) : 0x01010101u;
    float4 gv;
    uint32_t c0, c1, c2, c3;
    const float l0 = token(rv.x, av.x, (mv & 0xFFu) != 0, wv.x, b, a, gv.x, c0);
    const float l1 = token(rv.y, av.y, (mv & 0xFF00u) != 0, wv.y, b, a, gv.y, c1);
    const float l2 = token(rv.z, av.z, (mv & 0xFF0000u) != 0, wv.z, b, a, gv.z, c2);
    const float l3 = token(rv.w, av.w, (mv & 0xFF000000u) != 0, wv.w, b, a, gv.w, c3);
    a.add((l0 + l1) + (l2 + l3));
    if (grad) reinterpret_cast<float4*>(grad)[i] = gv;
    if (clip_mask) reinterpret_cast<uint32_t*>(clip_mask)[i] = c0 | (c1 << 8) | (c2 << 16) | (c3 << 24);
  }
  for (int64_t t = T4 * 4 + tid; t < T; t += stride) {
    float g;
    uint32_t cm;
    a.add(token(r[t], adv[t], mask ? mask[t] != 0 : true, wts ? wts[t] : 1.f, b, a, g, cm));
    if (grad) grad[t] = g;
    if (clip_mask) clip_mask[t] = static_cast<uint8_t>(cm);
  }
  const double loss = block_sum(static_cast<double>(a.s) + static_cast<double>(a.c), sh_d);
  const unsigned long long n_pos = block_sum<unsigned long long>(a.n_pos, sh_u);
  const unsigned long long n_neg = block_sum<unsigned long long>(a.n_neg, sh_u);
  const unsigned long long c_pos = block_sum<unsigned long long>(a.c_pos, sh_u);
  const unsigned long long c_neg = block_sum<unsigned long long>(a.c_neg, sh_u);
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
  if (!last) return;
  // The last block reduces the partials: thread i takes partials i, i + 256,
  // ... in order, then the fixed-order block sum.
  __threadfence();
  double L = 0.0;
  unsigned long long np = 0, nn = 0, cp = 0, cn = 0;
  for (unsigned k = threadIdx.x; k < gridDim.x; k += kThreads) {
    const volatile Partial& p = w->part[k];
    L += p.loss;
    np += p.n_pos;
    nn += p.n_neg;
    cp += p.c_pos;
    cn += p.c_neg;
  }
  L = block_sum(L, sh_d);
  np = block_sum(np, sh_u);
  nn = block_sum(nn, sh_u);
  cp = block_sum(cp, sh_u);
  cn = block_sum(cn, sh_u);
  if (threadIdx.x == 0) {
    fp8rl_clip_stats s;
    s.loss_sum = L;
    s.loss = n_valid ? L / static_cast<double>(n_valid) : 0.0;
    s.n_valid = static_cast<int64_t>(n_valid);
    s.n_pos = static_cast<int64_t>(np);
    s.n_neg = static_cast<int64_t>(nn);
    s.clipped_pos = static_cast<int64_t>(cp);
    s.clipped_neg = static_cast<int64_t>(cn);
    s.lo = b.lo;
    s.hi = b.hi;
    s.flags = n_valid ? 0 : 1;
    s.n_seq_valid = 0;
    *stats = s;
  }
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

// ------------------------------------------------------------ sequence mean
struct SeqWork {
  unsigned long long n_valid;
  unsigned int ticket;
  unsigned int n_seq_valid;
  unsigned int ticket2;
  unsigned int pad[59];
  Partial part[1];  // [grid]; the per-sequence counts follow the partials
};

size_t seq_counts_offset(int64_t T) {
  return align_up(sizeof(SeqWork) + sizeof(Partial) * static_cast<size_t>(grid_of(T)), 256);
}

// n_i per sequence, n_valid and S = #{i : n_i > 0} (counted by the atomics
// that find a sequence's count still zero).  Each
// warp walks its own contiguous range of tokens 32 at a time and carries the
// count of the sequence it is in across steps (responses are usually
// contiguous), so a sequence costs one atomic per warp that touches it rather
// than one per step.  Tokens with an id outside [0, n_seq) flag bad input and
// count nowhere.
__global__ void __launch_bounds__(kThreads) seq_count_kernel(const uint8_t* __restrict__ mask,
                                                             const int32_t* __restrict__ sid,
                                                             int64_t T, int64_t n_seq,
                                                             unsigned int* __restrict__ cnt,
                                                             SeqWork* w) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  const int64_t wid = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5);
  const int64_t per = ((T + nwarps - 1) / nwarps + 127) / 128 * 128;
  const int64_t beg = wid * per, end = min(T, beg + per);
  uint32_t nv = 0;
  bool bad = false;
  int cur_id = -1;        // warp-uniform: the sequence being counted and its count
  unsigned cur_cnt = 0;
  unsigned s_new = 0;     // lane 0: sequences this warp found empty
  for (int64_t base = beg; base < end; base += 128) {
    // four steps of 32 tokens: all loads issued before any is used
    int idv[4];
    bool on[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t t = base + u * 32 + lane;
      idv[u] = t < end ? __ldg(sid + t) : -1;
      on[u] = t < end && (!mask || __ldg(mask + t) != 0);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      // runs of equal (raw) ids among the 32 tokens, in lane order; masked
      // tokens keep their id, so padding inside a response does not split its
      // run, and each run adds the number of its valid tokens
      const int id = idv[u];
      const bool in_range = id >= 0 && id < n_seq;
      const bool valid = on[u] && in_range;
      if (base + u * 32 + lane < end && !in_range) bad = true;  // masked tokens too
      nv += valid;
      const unsigned vbits = __ballot_sync(0xffffffffu, valid);
      const int prev = __shfl_up_sync(0xffffffffu, id, 1);
      unsigned heads = __ballot_sync(0xffffffffu, lane == 0 || id != prev);
      while (heads) {
        const int h = __ffs(heads) - 1;
        heads &= heads - 1;
        const int next = heads ? __ffs(heads) - 1 : 32;
        const unsigned run = (next == 32 ? 0xffffffffu : ((1u << next) - 1u)) & ~((1u << h) - 1u);
        const unsigned n = __popc(vbits & run);
        if (n == 0) continue;  // no valid token in this run
        const int run_id = __shfl_sync(0xffffffffu, id, h);
        if (run_id == cur_id) {
          cur_cnt += n;
        } else {
          if (cur_id >= 0 && lane == 0) s_new += atomicAdd(&cnt[cur_id], cur_cnt) == 0u;
          cur_id = run_id;
          cur_cnt = n;
        }
      }
    }
  }
  if (cur_id >= 0 && lane == 0) s_new += atomicAdd(&cnt[cur_id], cur_cnt) == 0u;
  if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(&d_status, kErrDevice);
  const uint32_t s = __reduce_add_sync(0xffffffffu, nv);
  if (lane == 0 && s) atomicAdd(&w->n_valid, static_cast<unsigned long long>(s));
  // S: the atomics that found a sequence's count still zero
  if (lane == 0 && s_new) atomicAdd(&w->n_seq_valid, s_new);
}

__global__ void __launch_bounds__(kThreads) seq_surrogate_kernel(
    const float* __restrict__ r, const float* __restrict__ adv, const uint8_t* __restrict__ mask,
    const float* __restrict__ wts, const int32_t* __restrict__ sid, int64_t T, int64_t n_seq,
    const unsigned int* __restrict__ cnt, float lo_arg, float hi_arg, const float* __restrict__ bounds,
    float* __restrict__ grad, uint8_t* __restrict__ clip_mask, fp8rl_clip_stats* __restrict__ stats,
    SeqWork* w, bool vec) {
  __shared__ double sh_d[kThreads / 32];
  __shared__ unsigned long long sh_u[kThreads / 32];
  __shared__ bool last;
  Bounds b;
  b.lo = bounds ? bounds[0] : lo_arg;
  b.hi = bounds ? bounds[1] : hi_arg;
  const unsigned int S = w->n_seq_valid;
  const float inv_s = S ? 1.0f / static_cast<float>(S) : 0.f;
  Acc a;
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  // one token: 1/n_i (correctly rounded) scales its term, and 1/(S n_i) its gradient
  auto one = [&](float rt, float at, bool present, float wt, int id, float& g, uint32_t& cm) {
    const bool valid = present && id >= 0 && id < n_seq;
    const float inv_ni = valid ? __frcp_rn(static_cast<float>(__ldg(cnt + id))) : 1.f;
    b.inv_n = inv_s * inv_ni;
    a.add(token(rt, at, valid, wt, b, a, g, cm) * inv_ni);
  };
  const int64_t T4 = vec ? T / 4 : 0;
  for (int64_t i = tid; i < T4; i += stride) {
    const float4 rv = __ldg(reinterpret_cast<const float4*>(r) + i);
    const float4 av = __ldg(reinterpret_cast<const float4*>(adv) + i);
    const int4 iv = __ldg(reinterpret_cast<const int4*>(sid) + i);
    const float4 wv = wts ? __ldg(reinterpret_cast<const float4*>(wts) + i) : make_float4(1.f, 1.f, 1.f, 1.f);
    const uint32_t mv = mask ? __ldg(reinterpret_cast<const uint32_t*>(mask) + i) : 0x01010101u;
    float4 gv;
    uint32_t c0, c1, c2, c3;
    one(rv.x, av.x, (mv & 0xFFu) != 0, wv.x, iv.x, gv.x, c0);
    one(rv.y, av.y, (mv & 0xFF00u) != 0, wv.y, iv.y, gv.y, c1);
    one(rv.z, av.z, (mv & 0xFF0000u) != 0, wv.z, iv.z, gv.z, c2);
    one(rv.w, av.w, (mv & 0xFF000000u) != 0, wv.w, iv.w, gv.w, c3);
    if (grad) reinterpret_cast<float4*>(grad)[i] = gv;
    if (clip_mask) reinterpret_cast<uint32_t*>(clip_mask)[i] = c0 | (c1 << 8) | (c2 << 16) | (c3 << 24);
  }
  for (int64_t t = T4 * 4 + tid; t < T; t += stride) {
    float g;
    uint32_t cm;
    one(r[t], adv[t], mask ? mask[t] != 0 : true, wts ? wts[t] : 1.f, sid[t], g, cm);
    if (grad) grad[t] = g;
    if (clip_mask) clip_mask[t] = static_cast<uint8_t>(cm);
  }
  const double loss = block_sum(static_cast<double>(a.s) + static_cast<double>(a.c), sh_d);
  const unsigned long long n_pos = block_sum<unsigned long long>(a.n_pos, sh_u);
  const unsigned long long n_neg = block_sum<unsigned long long>(a.n_neg, sh_u);
  const unsigned long long c_pos = block_sum<unsigned long long>(a.c_pos, sh_u);
  const unsigned long long c_neg = block_sum<unsigned long long>(a.c_neg, sh_u);
  if (threadIdx.x == 0) {
    Partial& p = w->part[blockIdx.x];
    p.loss = loss;
    p.n_pos = n_pos;
    p.n_neg = n_neg;
    p.c_pos = c_pos;
    p.c_neg = c_neg;
    __threadfence();
    last = atomicAdd(&w->ticket2, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  double L = 0.0;
  unsigned long long np = 0, nn = 0, cp = 0, cn = 0;
  for (unsigned k = threadIdx.x; k < gridDim.x; k += kThreads) {
    const volatile Partial& p = w->part[k];
    L += p.loss;
    np += p.n_pos;
    nn += p.n_neg;
    cp += p.c_pos;
    cn += p.c_neg;
  }
  L = block_sum(L, sh_d);
  np = block_sum(np, sh_u);
  nn = block_sum(nn, sh_u);
  cp = block_sum(cp, sh_u);
  cn = block_sum(cn, sh_u);
  if (threadIdx.x == 0) {
    const unsigned long long n_valid = w->n_valid;
    fp8rl_clip_stats s;
    s.loss_sum = L;
    s.loss = S ? L / static_cast<double>(S) : 0.0;
    s.n_valid = static_cast<int64_t>(n_valid);
    s.n_pos = static_cast<int64_t>(np);
    s.n_neg = static_cast<int64_t>(nn);
    s.clipped_pos = static_cast<int64_t>(cp);
    s.clipped_neg = static_cast<int64_t>(cn);
    s.lo = b.lo;
    s.hi = b.hi;
    s.flags = n_valid ? 0 : 1;
    s.n_seq_valid = static_cast<int32_t>(S);
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
  if (mask) count_valid_kernel<<<grid, kThreads, 0, s>>>(mask, T, work);
  const bool vec = aligned(r, 16) && aligned(adv, 16) && aligned(w, 16) && aligned(grad, 16) &&
                   aligned(mask, 4) && aligned(clip_mask, 4);
  surrogate_kernel<<<grid, kThreads, 0, s>>>(r, adv, mask, w, T, lo, hi, bounds, grad, clip_mask,
                                              stats, work, vec);
  return cudaGetLastError();
}

size_t seq_surrogate_workspace_bytes(int64_t T, int64_t n_seq) {
  return seq_counts_offset(T) + align_up(static_cast<size_t>(n_seq > 0 ? n_seq : 1) * 4, 256);
}

cudaError_t launch_seq_surrogate(const float* r, const float* adv, const uint8_t* mask,
                                 const float* w, const int32_t* sid, int64_t n_seq, int64_t T,
                                 float lo, float hi, const float* bounds, float* grad,
                                 uint8_t* clip_mask, fp8rl_clip_stats* stats, void* ws,
                                 cudaStream_t s) {
  SeqWork* work = static_cast<SeqWork*>(ws);
  unsigned int* cnt = reinterpret_cast<unsigned int*>(static_cast<char*>(ws) + seq_counts_offset(T));
  cudaError_t e = cudaMemsetAsync(work, 0, sizeof(SeqWork), s);
  if (e == cudaSuccess && n_seq > 0) e = cudaMemsetAsync(cnt, 0, static_cast<size_t>(n_seq) * 4, s);
  if (e != cudaSuccess) return e;
  const int grid = grid_of(T);
  seq_count_kernel<<<grid, kThreads, 0, s>>>(mask, sid, T, n_seq, cnt, work);
  const bool vec = aligned(r, 16) && aligned(adv, 16) && aligned(sid, 16) && aligned(w, 16) &&
                   aligned(grad, 16) && aligned(mask, 4) && aligned(clip_mask, 4);
  seq_surrogate_kernel<<<grid, kThreads, 0, s>>>(r, adv, mask, w, sid, T, n_seq, cnt, lo, hi, bounds,
                                                  grad, clip_mask, stats, work, vec);
  return cudaGetLastError();
}

uint32_t loss_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
