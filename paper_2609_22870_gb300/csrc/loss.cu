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
// a mask, or when the caller passes the count, e.g. the calibration's, which
// reads the same mask), then the fused per-token pass writing g and the clip mask, four
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
//
// Sequence-level ratio clipping (the response-level trust region of the
// related-work discussion, §6): one ratio per response, the geometric mean of
// its token ratios s_i = exp((1/n_i) sum_t d_t), d_t = logp_t - logp_old_t,
// clipped like a token ratio with the response's advantage A_i:
//   loss = (1/S) sum_i -A_i m_i,  m_i = min(s_i, H) (A_i >= 0) / max(s_i, L),
//   g_t  = -A_i s_i / (n_i S) on valid tokens of unclipped responses.
// The exponent sums are exact integers: each d_t (|d_t| <= 128) is taken to
// the 2^-32 grid (exact for |d_t| >= 2^-8, where d_t 2^32 is already an
// integer) and summed with 64-bit integer atomics, so the result does not
// depend on the order of the tokens or of the atomics.
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

// The launch grid of a kernel whose CTAs each take an equal share of the
// work: `grid` (what the workspace was sized for) capped at one full wave of
// the CTAs the SMs hold at once, so no CTA waits for a second wave.
template <typename Kernel>
int wave_grid(Kernel* kernel, int grid) {
  const int cap = sm_count() * min(kCtasPerSm, resident_ctas(reinterpret_cast<const void*>(kernel), kThreads));
  return grid < cap ? grid : cap;
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
  int64_t i = tid;
  // four 16-byte loads in flight per thread, then the remainder one at a time
  for (; i + 3 * stride < T16; i += 4 * stride) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = __ldg(reinterpret_cast<const uint4*>(mask) + i + u * stride);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      n += nonzero_bytes(v[u].x) + nonzero_bytes(v[u].y) + nonzero_bytes(v[u].z) + nonzero_bytes(v[u].w);
  }
  for (; i < T16; i += stride) {
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

// Clip fractions of §3 (PPO's clip fraction, split by advantage sign): the
// share of A > 0 units clipped at H, of A < 0 units clipped at L, and of all
// valid units clipped; 0 where the denominator is 0.  Units are tokens for the
// token-level calls and responses for sequence-level clipping.
__device__ __forceinline__ void set_clip_fractions(fp8rl_clip_stats& s, unsigned long long n_all) {
  s.clip_frac_pos = s.n_pos ? static_cast<double>(s.clipped_pos) / static_cast<double>(s.n_pos) : 0.0;
  s.clip_frac_neg = s.n_neg ? static_cast<double>(s.clipped_neg) / static_cast<double>(s.n_neg) : 0.0;
  s.clip_frac = n_all ? static_cast<double>(s.clipped_pos + s.clipped_neg) / static_cast<double>(n_all) : 0.0;
}

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
    fp8rl_clip_stats* __restrict__ stats, Work* w, const int64_t* __restrict__ nv_in, bool vec) {
  __shared__ double sh_d[kThreads / 32];
  __shared__ unsigned long long sh_u[kThreads / 32];
  __shared__ bool last;
  Bounds b;
  b.lo = bounds ? bounds[0] : lo_arg;
  b.hi = bounds ? bounds[1] : hi_arg;
  const unsigned long long n_valid =
      !mask ? static_cast<unsigned long long>(T)
            : (nv_in ? static_cast<unsigned long long>(*nv_in) : w->n_valid);
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
    set_clip_fractions(s, n_valid);
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
    set_clip_fractions(s, n_valid);
    *stats = s;
  }
}

// ------------------------------------------------------------ sequence-level ratio
constexpr float kSeqLvlDMax = 128.f;  // largest |d_t| of a valid token

struct SeqLvlWork {
  unsigned long long n_valid;
  unsigned int n_seq_valid;
  unsigned int ticket;
  unsigned int pad[60];
  // then: q[n_seq] (int64 fixed-point exponent sums), cnt[n_seq] (uint32),
  // part[grid of the sequence pass], coef[n_seq] (float)
};

struct SeqLvlLayout {
  size_t q, cnt, part, coef, zero_bytes, total;
};

int seq_grid_of(int64_t n_seq) {
  const int64_t want = (n_seq + kThreads - 1) / kThreads;
  const int64_t cap = static_cast<int64_t>(sm_count()) * kCtasPerSm;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

SeqLvlLayout seq_lvl_layout(int64_t n_seq) {
  const size_t n = static_cast<size_t>(n_seq > 0 ? n_seq : 1);
  SeqLvlLayout l;
  l.q = sizeof(SeqLvlWork);
  l.cnt = l.q + 8 * n;
  l.zero_bytes = l.cnt + 4 * n;  // header, q and cnt are zeroed every call
  l.part = align_up(l.zero_bytes, 256);
  l.coef = align_up(l.part + sizeof(Partial) * static_cast<size_t>(seq_grid_of(n_seq)), 256);
  l.total = align_up(l.coef + 4 * n, 256);
  return l;
}

// Pass 1: per sequence the valid-token count n_i and the fixed-point sum
// Q_i = sum_t RNE(d_t 2^32), plus S = #{i : n_i > 0}.  Each warp walks its
// own contiguous range, 128 tokens a step (four consecutive tokens a lane).
// Every lane accumulates the tokens of the warp's current sequence in
// registers; only a step that holds a valid token of another sequence (a
// response boundary) makes the warp cooperate: it flushes the current
// sequence (warp sum, one pair of atomics), takes the step's last valid id as
// the new current sequence, and sends any other token (a response shorter
// than a step, or ids in no order) straight to the atomics.  Invalid tokens
// add nothing whatever their id.  Without SUMS only the counts are formed (the
// sequence-mean surrogate's count pass).
template <bool VEC, bool SUMS, typename WorkT>
__global__ void __launch_bounds__(kThreads) seq_accum_kernel(
    const float* __restrict__ logp, const float* __restrict__ logp_old,
    const uint8_t* __restrict__ mask, const int32_t* __restrict__ sid, int64_t T, int64_t n_seq,
    unsigned long long* __restrict__ qsum, unsigned int* __restrict__ cnt, WorkT* w) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  const int64_t wid = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5);
  const int64_t per = ((T + nwarps - 1) / nwarps + 127) / 128 * 128;
  const int64_t beg = wid * per, end = min(T, beg + per);
  uint32_t nv = 0, s_new = 0;
  bool bad = false;
  int cur = -1;  // warp-uniform current sequence
  long long acc_q = 0;
  unsigned acc_n = 0;
  auto flush = [&]() {
    long long q = acc_q;
    if (SUMS) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    }
    const unsigned n = __reduce_add_sync(0xffffffffu, acc_n);
    if (lane == 0 && n) {
      s_new += atomicAdd(&cnt[cur], n) == 0u;
      if (SUMS) atomicAdd(&qsum[cur], static_cast<unsigned long long>(q));
    }
    acc_q = 0;
    acc_n = 0;
  };
  // one 128-token step (four consecutive tokens a lane), after its loads
  auto step = [&](const int (&id)[4], const float (&lp)[4], const float (&lo)[4], const bool (&on)[4], int64_t t0) {
    long long q[4];
    bool v[4];
    bool match = true;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const bool in_range = id[k] >= 0 && id[k] < n_seq;
      if (t0 + k < end && !in_range) bad = true;  // masked tokens too
      v[k] = on[k] && in_range;
      float d = lp[k] - lo[k];
      if (SUMS && v[k] && !(fabsf(d) <= kSeqLvlDMax)) {  // out of range or NaN
        bad = true;
        d = d != d ? 0.f : fminf(fmaxf(d, -kSeqLvlDMax), kSeqLvlDMax);
      }
      // d 2^32 is exact in float32; the conversion rounds to nearest even
      q[k] = SUMS && v[k] ? __float2ll_rn(d * 4294967296.0f) : 0ll;
      nv += v[k];
      match = match && (!v[k] || id[k] == cur);
    }
    if (__all_sync(0xffffffffu, match)) {  // the step continues the current sequence
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        acc_q += q[k];
        acc_n += v[k];
      }
      return;
    }
    // a boundary: finish the current sequence with this step's tokens of it
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (v[k] && id[k] == cur) {
        acc_q += q[k];
        acc_n += 1;
        v[k] = false;
      }
    flush();
    // the step's last valid token names the sequence that may run on
    int last_id = -1;
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (v[k]) last_id = id[k];
    const unsigned has = __ballot_sync(0xffffffffu, last_id >= 0);
    if (has) cur = __shfl_sync(0xffffffffu, last_id, 31 - __clz(has));
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (v[k] && id[k] == cur) {
        acc_q += q[k];
        acc_n += 1;
        v[k] = false;
      }
    // whatever is left belongs to neither: one pair of atomics per token
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (v[k]) {
        s_new += atomicAdd(&cnt[id[k]], 1u) == 0u;
        if (SUMS) atomicAdd(&qsum[id[k]], static_cast<unsigned long long>(q[k]));
      }
  };
  auto load_vec = [&](int64_t t0, int (&id)[4], float (&lp)[4], float (&lo)[4], bool (&on)[4]) {
    const int4 iv = __ldg(reinterpret_cast<const int4*>(sid + t0));
    const uint32_t mv = mask ? __ldg(reinterpret_cast<const uint32_t*>(mask + t0)) : 0x01010101u;
    id[0] = iv.x, id[1] = iv.y, id[2] = iv.z, id[3] = iv.w;
    if (SUMS) {
      const float4 a = __ldg(reinterpret_cast<const float4*>(logp + t0));
      const float4 b = __ldg(reinterpret_cast<const float4*>(logp_old + t0));
      lp[0] = a.x, lp[1] = a.y, lp[2] = a.z, lp[3] = a.w;
      lo[0] = b.x, lo[1] = b.y, lo[2] = b.z, lo[3] = b.w;
    } else {
#pragma unroll
      for (int k = 0; k < 4; ++k) lp[k] = lo[k] = 0.f;
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) on[k] = ((mv >> (8 * k)) & 0xFFu) != 0;
  };
  int64_t base = beg;
  // without the sums a step loads only ids and mask (5 B a token): four full
  // steps' loads in flight before any is processed
  if (VEC && !SUMS) {
    for (; base + 511 < end; base += 512) {
      int id[4][4];
      float lp[4][4], lo[4][4];
      bool on[4][4];
#pragma unroll
      for (int k = 0; k < 4; ++k) load_vec(base + 128 * k + 4 * lane, id[k], lp[k], lo[k], on[k]);
#pragma unroll
      for (int k = 0; k < 4; ++k) step(id[k], lp[k], lo[k], on[k], base + 128 * k + 4 * lane);
    }
  }
  // two full steps' loads in flight before either is processed
  if (VEC) {
    for (; base + 255 < end; base += 256) {
      int idA[4], idB[4];
      float lpA[4], loA[4], lpB[4], loB[4];
      bool onA[4], onB[4];
      load_vec(base + 4 * lane, idA, lpA, loA, onA);
      load_vec(base + 128 + 4 * lane, idB, lpB, loB, onB);
      step(idA, lpA, loA, onA, base + 4 * lane);
      step(idB, lpB, loB, onB, base + 128 + 4 * lane);
    }
  }
  for (; base < end; base += 128) {
    const int64_t t0 = base + 4 * lane;
    int id[4];
    float lp[4], lo[4];
    bool on[4];
    if (VEC && t0 + 3 < end) {
      load_vec(t0, id, lp, lo, on);
    } else {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int64_t t = t0 + k;
        const bool in = t < end;
        id[k] = in ? __ldg(sid + t) : 0;
        lp[k] = SUMS && in ? __ldg(logp + t) : 0.f;
        lo[k] = SUMS && in ? __ldg(logp_old + t) : 0.f;
        on[k] = in && (!mask || __ldg(mask + t) != 0);
        if (!in) id[k] = cur;  // past the end: nothing to add
      }
    }
    step(id, lp, lo, on, t0);
  }
  flush();
  if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(&d_status, kErrDevice);
  const uint32_t sv = __reduce_add_sync(0xffffffffu, nv);
  const uint32_t sn = __reduce_add_sync(0xffffffffu, s_new);
  if (lane == 0 && sv) atomicAdd(&w->n_valid, static_cast<unsigned long long>(sv));
  if (lane == 0 && sn) atomicAdd(&w->n_seq_valid, sn);
}

// Pass 2, one thread per sequence: s_i = fl32(exp(Q_i 2^-32 / n_i)), the clip
// bits, the term -A_i m_i (an exact float64 product) and the gradient
// coefficient fl32(-A_i s_i / (n_i S)) of its valid tokens; the terms meet in
// a fixed-order reduction (last block), which also writes the statistics.
__global__ void __launch_bounds__(kThreads) seq_lvl_seq_kernel(
    const float* __restrict__ adv_seq, int64_t n_seq, const unsigned long long* __restrict__ qsum,
    const unsigned int* __restrict__ cnt, float lo_arg, float hi_arg, const float* __restrict__ bounds,
    float* __restrict__ seq_ratio, uint8_t* __restrict__ seq_clip, float* __restrict__ coef,
    Partial* __restrict__ part, fp8rl_clip_stats* __restrict__ stats, SeqLvlWork* w) {
  __shared__ double sh_d[kThreads / 32];
  __shared__ unsigned long long sh_u[kThreads / 32];
  __shared__ bool last;
  const float lo = bounds ? bounds[0] : lo_arg;
  const float hi = bounds ? bounds[1] : hi_arg;
  const unsigned int S = w->n_seq_valid;
  double L = 0.0;
  uint32_t np = 0, nn = 0, cp = 0, cn = 0;
  for (int64_t i = blockIdx.x * (int64_t)kThreads + threadIdx.x; i < n_seq;
       i += (int64_t)gridDim.x * kThreads) {
    const unsigned n = cnt[i];
    float s = 0.f, c = 0.f;
    uint32_t cm = 0;
    if (n) {
      const double mu = static_cast<double>(static_cast<long long>(qsum[i])) * 0x1p-32 /
                        static_cast<double>(n);
      s = static_cast<float>(exp(mu));
      const float A = adv_seq[i];
      const bool up = A > 0.f && s >= hi;
      const bool dn = A < 0.f && s <= lo;
      const float m = A >= 0.f ? fminf(s, hi) : fmaxf(s, lo);
      L += -static_cast<double>(A) * static_cast<double>(m);
      np += A > 0.f;
      nn += A < 0.f;
      cp += up;
      cn += dn;
      cm = (up ? FP8RL_CLIP_HI : 0u) | (dn ? FP8RL_CLIP_LO : 0u);
      if (!(up || dn))
        c = static_cast<float>(-static_cast<double>(A) * static_cast<double>(s) /
                               (static_cast<double>(n) * static_cast<double>(S)));
    }
    coef[i] = c;
    if (seq_ratio) seq_ratio[i] = s;
    if (seq_clip) seq_clip[i] = static_cast<uint8_t>(cm);
  }
  L = block_sum(L, sh_d);
  const unsigned long long bnp = block_sum<unsigned long long>(np, sh_u);
  const unsigned long long bnn = block_sum<unsigned long long>(nn, sh_u);
  const unsigned long long bcp = block_sum<unsigned long long>(cp, sh_u);
  const unsigned long long bcn = block_sum<unsigned long long>(cn, sh_u);
  if (threadIdx.x == 0) {
    Partial& p = part[blockIdx.x];
    p.loss = L;
    p.n_pos = bnp;
    p.n_neg = bnn;
    p.c_pos = bcp;
    p.c_neg = bcn;
    __threadfence();
    last = atomicAdd(&w->ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  double tl = 0.0;
  unsigned long long tnp = 0, tnn = 0, tcp = 0, tcn = 0;
  for (unsigned k = threadIdx.x; k < gridDim.x; k += kThreads) {
    const volatile Partial& p = part[k];
    tl += p.loss;
    tnp += p.n_pos;
    tnn += p.n_neg;
    tcp += p.c_pos;
    tcn += p.c_neg;
  }
  tl = block_sum(tl, sh_d);
  tnp = block_sum(tnp, sh_u);
  tnn = block_sum(tnn, sh_u);
  tcp = block_sum(tcp, sh_u);
  tcn = block_sum(tcn, sh_u);
  if (threadIdx.x == 0) {
    const unsigned long long n_valid = w->n_valid;
    fp8rl_clip_stats st;
    st.loss_sum = tl;
    st.loss = S ? tl / static_cast<double>(S) : 0.0;
    st.n_valid = static_cast<int64_t>(n_valid);
    st.n_pos = static_cast<int64_t>(tnp);
    st.n_neg = static_cast<int64_t>(tnn);
    st.clipped_pos = static_cast<int64_t>(tcp);
    st.clipped_neg = static_cast<int64_t>(tcn);
    st.lo = lo;
    st.hi = hi;
    st.flags = n_valid ? 0 : 1;
    st.n_seq_valid = static_cast<int32_t>(S);
    set_clip_fractions(st, S);  // over responses
    *stats = st;
  }
}

// Pass 3: g_t = coef[seq(t)] on valid tokens, 0 elsewhere; four tokens per
// thread and step with 16-byte loads and stores when the arrays allow.
__global__ void __launch_bounds__(kThreads) seq_lvl_grad_kernel(
    const uint8_t* __restrict__ mask, const int32_t* __restrict__ sid, int64_t T, int64_t n_seq,
    const float* __restrict__ coef, float* __restrict__ grad, bool vec) {
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  auto one = [&](int id, bool present) {
    return present && id >= 0 && id < n_seq ? __ldg(coef + id) : 0.f;
  };
  const int64_t T4 = vec ? T / 4 : 0;
  for (int64_t i = tid; i < T4; i += stride) {
    const int4 iv = __ldg(reinterpret_cast<const int4*>(sid) + i);
    const uint32_t mv = mask ? __ldg(reinterpret_cast<const uint32_t*>(mask) + i) : 0x01010101u;
    float4 g;
    g.x = one(iv.x, (mv & 0xFFu) != 0);
    g.y = one(iv.y, (mv & 0xFF00u) != 0);
    g.z = one(iv.z, (mv & 0xFF0000u) != 0);
    g.w = one(iv.w, (mv & 0xFF000000u) != 0);
    reinterpret_cast<float4*>(grad)[i] = g;
  }
  for (int64_t t = T4 * 4 + tid; t < T; t += stride) grad[t] = one(sid[t], mask ? mask[t] != 0 : true);
}

}  // namespace

size_t surrogate_workspace_bytes(int64_t T) {
  return align_up(sizeof(Work) + sizeof(Partial) * static_cast<size_t>(grid_of(T)), 256);
}

cudaError_t launch_surrogate(const float* r, const float* adv, const uint8_t* mask,
                             const float* w, int64_t T, float lo, float hi, const float* bounds,
                             const int64_t* n_valid, float* grad, uint8_t* clip_mask,
                             fp8rl_clip_stats* stats, void* ws, cudaStream_t s) {
  Work* work = static_cast<Work*>(ws);
  cudaError_t e = cudaMemsetAsync(work, 0, sizeof(Work), s);
  if (e != cudaSuccess) return e;
  const int grid = wave_grid(surrogate_kernel, grid_of(T));
  if (mask && !n_valid) count_valid_kernel<<<wave_grid(count_valid_kernel, grid_of(T)), kThreads, 0, s>>>(mask, T, work);
  const bool vec = aligned(r, 16) && aligned(adv, 16) && aligned(w, 16) && aligned(grad, 16) &&
                   aligned(mask, 4) && aligned(clip_mask, 4);
  surrogate_kernel<<<grid, kThreads, 0, s>>>(r, adv, mask, w, T, lo, hi, bounds, grad, clip_mask,
                                              stats, work, n_valid, vec);
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
  const int grid = wave_grid(seq_surrogate_kernel, grid_of(T));
  if (aligned(sid, 16) && aligned(mask, 4))
    seq_accum_kernel<true, false><<<wave_grid(seq_accum_kernel<true, false, SeqWork>, grid_of(T)), kThreads, 0, s>>>(
        nullptr, nullptr, mask, sid, T, n_seq, nullptr, cnt, work);
  else
    seq_accum_kernel<false, false><<<wave_grid(seq_accum_kernel<false, false, SeqWork>, grid_of(T)), kThreads, 0, s>>>(
        nullptr, nullptr, mask, sid, T, n_seq, nullptr, cnt, work);
  const bool vec = aligned(r, 16) && aligned(adv, 16) && aligned(sid, 16) && aligned(w, 16) &&
                   aligned(grad, 16) && aligned(mask, 4) && aligned(clip_mask, 4);
  seq_surrogate_kernel<<<grid, kThreads, 0, s>>>(r, adv, mask, w, sid, T, n_seq, cnt, lo, hi, bounds,
                                                  grad, clip_mask, stats, work, vec);
  return cudaGetLastError();
}

size_t seq_level_workspace_bytes(int64_t, int64_t n_seq) { return seq_lvl_layout(n_seq).total; }

cudaError_t launch_seq_level(const float* logp, const float* logp_old, const float* adv_seq,
                             const uint8_t* mask, const int32_t* sid, int64_t n_seq, int64_t T,
                             float lo, float hi, const float* bounds, float* seq_ratio,
                             uint8_t* seq_clip, float* grad, fp8rl_clip_stats* stats, void* ws,
                             cudaStream_t s) {
  const SeqLvlLayout l = seq_lvl_layout(n_seq);
  char* base = static_cast<char*>(ws);
  SeqLvlWork* work = reinterpret_cast<SeqLvlWork*>(base);
  auto* q = reinterpret_cast<unsigned long long*>(base + l.q);
  auto* cnt = reinterpret_cast<unsigned int*>(base + l.cnt);
  auto* part = reinterpret_cast<Partial*>(base + l.part);
  auto* coef = reinterpret_cast<float*>(base + l.coef);
  cudaError_t e = cudaMemsetAsync(base, 0, l.zero_bytes, s);
  if (e != cudaSuccess) return e;
  const bool vec4 = aligned(logp, 16) && aligned(logp_old, 16) && aligned(sid, 16) && aligned(mask, 4);
  if (vec4)
    seq_accum_kernel<true, true><<<wave_grid(seq_accum_kernel<true, true, SeqLvlWork>, grid_of(T)), kThreads, 0, s>>>(
        logp, logp_old, mask, sid, T, n_seq, q, cnt, work);
  else
    seq_accum_kernel<false, true><<<wave_grid(seq_accum_kernel<false, true, SeqLvlWork>, grid_of(T)), kThreads, 0, s>>>(
        logp, logp_old, mask, sid, T, n_seq, q, cnt, work);
  seq_lvl_seq_kernel<<<wave_grid(seq_lvl_seq_kernel, seq_grid_of(n_seq)), kThreads, 0, s>>>(adv_seq, n_seq, q, cnt, lo, hi, bounds,
                                                             seq_ratio, seq_clip, coef, part, stats, work);
  if (grad) {
    const bool vec = aligned(sid, 16) && aligned(grad, 16) && aligned(mask, 4);
    seq_lvl_grad_kernel<<<wave_grid(seq_lvl_grad_kernel, grid_of(T)), kThreads, 0, s>>>(mask, sid, T, n_seq, coef,
                                                                                     grad, vec);
  }
  return cudaGetLastError();
}

uint32_t loss_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
