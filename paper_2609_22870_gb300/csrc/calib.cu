// a5: Calibrated Clipping (§4, Eq. 5, Algorithm 1) on the GPU.
//
// Stage 1 (lower-bound alignment): k = #{A<0 : r_bf16 <= c_lo}; L* is the
// float32 threshold in I_L minimising |#{A<0 : r_fp8 <= L} - k|, nearest c_lo.
// Stage 2 (upper-bound rebalancing, Eq. 5): with e_t = (coef_t r_t) A_t
// rounded to integers q_t = RNE(e_t 2^s), N_bf, D_bf, D_fp8 are exact sums and
// H* is the float32 in I_H minimising |P(H) D_bf - N_bf D_fp8|,
// P(H) = sum_{A>0, r_fp8 < H} q, nearest c_hi.  Then SmoothUpdate.
//
// EXACT mode finds each optimum with a weighted radix select over the float32
// bit patterns of the ratios (non-negative floats order like their bits):
// three histogram passes (11, 11, 10 bits) locate the smallest ratio u whose
// cumulative weight crosses the target, one more pass finds u's neighbours and
// the pieces of the step function that contain the ends of the search
// interval, and a single-block decide step turns them into the bound.  Counts
// and fixed-point sums are integers, so every reduction order gives the same
// bits and the result is reproducible to the last bit.  GRID mode histograms
// the ratios over Algorithm 1's candidate thresholds instead.
//
// Passes are grid-stride kernels with shared-memory histograms flushed by
// atomics; decide steps run in one block of 1024 threads.
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace fp8rl {
namespace {

__device__ uint32_t d_status;

constexpr int kBuckets = 2048;
constexpr int kCoopThreads = 512;         // block of the one-launch (cooperative) kernel
constexpr int64_t kCoopMaxT = 1 << 18;    // tokens up to which one launch does it all
constexpr int kCoopTokensPerBlock = 2048; // its grid: ceil(T / 2048) blocks, at most 128
constexpr int kCoopMaxBlocks = 128;

constexpr unsigned kNone = 0xFFFFFFFFu;

enum Stage : int {
  kPrep = 0,    // counts, emax, input checks; L histogram digit 0 / L grid counts
  kSums = 1,    // N_bf, D_bf; L digit 1 (exact) | D_fp8, k_fp8, H grid sums (grid)
  kL2 = 2,      // L digit 2
  kLNb = 3,     // L neighbours
  kH0 = 4,      // D_fp8, k_fp8, H digit 0
  kH1 = 5,
  kH2 = 6,
  kHNb = 7,     // H neighbours
  kPFin = 8     // P(H*)
};

struct State {
  // accumulated by passes (zeroed before the first pass)
  unsigned long long n_neg, n_pos, k_bf16, k_fp8;
  unsigned long long emax_bits;  // frexp exponent of max|e| plus kEBias (0 = no term)
  unsigned long long s_pos_bf, s_neg_bf, s_neg_fp, s_pos_fp;  // int64 two's complement
  unsigned int bad;
  unsigned int bar_count, bar_gen;  // grid barrier of the one-launch kernel
  unsigned int nb_below1;  // 1 + max{key < u} (0 = none)
  unsigned int nb_above;   // min{key > u}     (kNone = none)
  unsigned int nb_mpiece;  // L: min{key > key(lo_min)}   H: min{key >= key(hi_min), q > 0}
  unsigned int nb_Mpiece1; // L: 1 + max{key <= key(lo_max)}   H: 1 + max{key < key(hi_max), q > 0}
  unsigned int pad0;
  // EXACT mode selects only among the ratios inside the search interval (the
  // others cannot move a bound inside it): the radix histograms count A<0
  // tokens with lo_min <= r_fp8 <= lo_max and weigh A>0 tokens with
  // hi_min <= r_fp8 < hi_max; what lies below enters the select as `below`
  unsigned long long l_below;  // #{A<0 : r_fp8 < lo_min}
  unsigned long long l_in;     // #{A<0 : lo_min <= r_fp8 <= lo_max}
  unsigned long long h_below;  // sum_{A>0, r_fp8 < hi_min} q_fp8 (int64 two's complement)
  // The tokens inside the intervals are also written to two lists (keys of
  // I_L's A<0 tokens from the first pass; keys and q_fp8 of I_H's A>0 tokens
  // from the H digit-0 pass), and the later selection passes read only the
  // lists.  What they would have met outside the intervals is kept here
  // (u32 maxima; a minimum is kept as the maximum of ~key, 0 = none):
  unsigned int l_nb_below1;     // 1 + max{key : A<0, r < lo_min}
  unsigned int l_nb_above_inv;  // ~min{key : A<0, r > lo_max}
  unsigned int l_mp_inv;        // ~min{key in I_L : key > key(lo_min)}
  unsigned int l_Mp1;           // 1 + max{key in I_L}
  unsigned int h_nb_below1;     // 1 + max{key : A>0, r < hi_min, q != 0}
  unsigned int h_nb_above_inv;  // ~min{key : A>0, r >= hi_max, q != 0}
  unsigned int h_top1;          // 1 + max{key : A>0, r >= hi_max, q != 0}
  unsigned int h_mp_inv;        // ~min{key in I_H : q != 0}
  unsigned int h_Mp1;           // 1 + max{key in I_H : q != 0}
  unsigned int pad2;
  unsigned long long n_valid;   // valid tokens (any advantage), for the surrogate's mean
  // written by decide steps
  int shift;
  int found;
  unsigned int prefix;
  unsigned int u_key;
  long long below;
  long long p_lt, p_le;
  unsigned long long tgt_hi, tgt_lo;  // X as unsigned 128-bit
  long long dmul;                     // D
  float lo_star, hi_star;
  int flags;
  int h_active;  // stage 2 runs (not degenerate)
  int p_known;   // P(H*) = s_pos_fp already known: the last pass is skipped
  int pad1;
  // histograms
  unsigned long long h_cnt[kBuckets];
  unsigned long long h_w[kBuckets];
};

struct Args {
  const float* r_fp8;
  const float* r_bf16;
  const float* adv;
  const uint8_t* mask;
  const float* coef;
  int64_t T;
  float c_lo, c_hi;
  float lo_min, lo_max, hi_min, hi_max;
  float delta_lo, delta_hi;
  float lo_old, hi_old;
  int grid_mode;
  double lo_grid0, hi_grid0, step;  // Algorithm 1 grids: fl32(x0 + i * step)
  int n_lcand, n_hcand;
  State* st;
  fp8rl_calib_result* out;
  // Interval lists (EXACT mode), one segment per warp of the full passes
  // (nseg segments of seg_cap entries, each warp's tokens fit its segment, so
  // no list entry needs an atomic), with the segment's fill in *_cnt[seg]:
  unsigned* l_keys;   // keys of the A<0 tokens inside I_L
  unsigned* l_cnt;
  unsigned* h_keys;   // keys of the A>0 tokens inside I_H
  long long* h_q;     // their q_fp8
  unsigned* h_cnt;
  unsigned nseg, seg_cap;
};

__device__ __forceinline__ void flag(uint32_t bits) { atomicOr(&d_status, bits); }

__device__ __forceinline__ unsigned key_of(float r) { return __float_as_uint(r) & 0x7FFFFFFFu; }

// ---- Eq. 5 terms in integer arithmetic (no float64 instruction per token).
// e = fl64(fl64(c r) a): c r is exact in float64 (48-bit significand); the
// product with a has up to 72 bits and the float64 multiply rounds it to 53,
// to nearest, ties to even.  Both roundings (to 53 bits, then to an integer
// at scale 2^s) are carried out on the exact integer significands.
constexpr int kEBias = 2048;  // exponents of max|e| are stored biased (0 = no term)

// |x| = m 2^e with an integer significand m < 2^24.
__device__ __forceinline__ void split(float x, unsigned& m, int& e) {
  const unsigned b = __float_as_uint(x) & 0x7FFFFFFFu;
  const unsigned ex = b >> 23, fx = b & 0x7FFFFFu;
  if (ex == 0) {
    m = fx;
    e = -149;
  } else {
    m = fx | 0x800000u;
    e = static_cast<int>(ex) - 150;
  }
}

// |fl64(fl64(c r) a)| = m 2^e with m < 2^53 (m = 0 for a zero product).
__device__ __forceinline__ void term53(float c, float r, float a, unsigned long long& m53, int& e53) {
  unsigned mc, mr, ma;
  int ec, er, ea;
  split(c, mc, ec);
  split(r, mr, er);
  split(a, ma, ea);
  const unsigned long long p = static_cast<unsigned long long>(mc) * mr;  // < 2^48
  const unsigned long long lo = p * ma;
  const unsigned long long hi = __umul64hi(p, static_cast<unsigned long long>(ma));  // < 2^8
  int e = ec + er + ea;
  if ((lo | hi) == 0) {
    m53 = 0;
    e53 = 0;
    return;
  }
  const int len = hi ? 128 - __clzll(static_cast<long long>(hi)) : 64 - __clzll(static_cast<long long>(lo));
  if (len <= 53) {
    m53 = lo;
    e53 = e;
    return;
  }
  const int d = len - 53;  // 1 .. 19
  unsigned long long m = (hi << (64 - d)) | (lo >> d);
  const unsigned long long rem = lo & ((1ull << d) - 1);
  const unsigned long long half = 1ull << (d - 1);
  if (rem > half || (rem == half && (m & 1))) ++m;
  e += d;
  if (m >> 53) {
    m >>= 1;
    ++e;
  }
  m53 = m;
  e53 = e;
}

// frexp exponent E of |fl64(fl64(c r) a)| (value in [2^(E-1), 2^E)) plus
// kEBias; 0 for a zero product.
__device__ __forceinline__ unsigned term_exponent(float c, float r, float a) {
  unsigned long long m;
  int e;
  term53(c, r, a, m, e);
  if (m == 0) return 0;
  return static_cast<unsigned>(64 - __clzll(static_cast<long long>(m)) + e + kEBias);
}

// q_t = RNE(fl64(fl64(c r) a) 2^s) as int64, on the exact integer significands.
__device__ __forceinline__ long long fixed_term_exact(float c, float r, float a, int s) {
  unsigned long long m;
  int e;
  term53(c, r, a, m, e);
  if (m == 0) return 0;
  const int t = e + s;
  unsigned long long q;
  if (t >= 0) {
    q = m << (t < 63 ? t : 63);
  } else {
    const int d = -t;
    if (d > 54) {
      q = 0;
    } else {
      q = m >> d;
      const unsigned long long rem = m & ((1ull << d) - 1);
      const unsigned long long half = 1ull << (d - 1);
      if (rem > half || (rem == half && (q & 1))) ++q;
    }
  }
  return a < 0.f ? -static_cast<long long>(q) : static_cast<long long>(q);
}

// The same q_t from float32 arithmetic wherever that decides it; false sends
// the token to fixed_term_exact.  With V = c r |a| 2^s (c, r >= 0):
//   hi + lo = c r exactly (lo = fma(c, r, -hi), exact for |hi| >= 2^-102),
//   p1 + e1 = hi |a| exactly (the same for |p1| >= 2^-102),
//   A = p1 2^s (exact: a power-of-two scale, s in [-126, 127]),
//   B = fl(e1 + fl(lo |a|)) 2^s, with A + B within 2^-46 |A| of V;
//   Ai = rint(A) and f = fl((A - Ai) + B) (A - Ai exact).
// For |A| < 2^35, Ai + f lies within 2^-11 + 2^-12 of V, and fl64(V) within
// 2^-53 |V| <= 2^-18 of V, so both are within 2^-10 of each other.  When f is
// more than 2^-9 from the nearest half-integer, no integer rounding boundary
// lies between them, and RNE(fl64(V)) = Ai + rint(f).  Ties, huge, tiny,
// zero and non-finite products take the exact path.
__device__ __forceinline__ bool fixed_term_fast(float c, float r, float a, int s, long long& q) {
  const float ca = fabsf(a);
  const float hi = c * r;
  const float p1 = hi * ca;
  if (!(hi >= 0x1p-102f && p1 >= 0x1p-102f) || s < -126 || s > 127) return false;
  const float lo = fmaf(c, r, -hi);
  const float e1 = fmaf(hi, ca, -p1);
  const float sc = __int_as_float((s + 127) << 23);
  const float A = p1 * sc;
  if (!(A < 0x1p35f)) return false;  // also catches an infinite product
  const float B = (e1 + lo * ca) * sc;
  const float Ai = rintf(A);
  const float f = (A - Ai) + B;
  const float fi = rintf(f);
  if (!(fabsf(fabsf(f - fi) - 0.5f) > 0x1p-9f)) return false;
  const long long m = static_cast<long long>(Ai) + static_cast<long long>(fi);
  q = a < 0.f ? -m : m;
  return true;
}

__device__ __forceinline__ long long fixed_term(float c, float r, float a, int s) {
  long long q;
  if (fixed_term_fast(c, r, a, s, q)) return q;
  return fixed_term_exact(c, r, a, s);
}

__device__ __forceinline__ bool digit_match(unsigned key, int digit, unsigned prefix) {
  if (digit == 0) return true;
  if (digit == 1) return (key >> 21) == prefix;
  return (key >> 10) == prefix;
}

__device__ __forceinline__ unsigned digit_of(unsigned key, int digit) {
  if (digit == 0) return key >> 21;
  if (digit == 1) return (key >> 10) & 0x7FFu;
  return key & 0x3FFu;
}

// frexp exponent of |fl64(fl64(c r) a)| plus kEBias (0 for a zero product),
// from the float32 product wherever that settles it: the two float32
// roundings leave it within a factor 1 +- 2^-22 of the exact product, so when
// its significand lies at least 8 ulps (2^-20) from both ends of its binade
// the exact product shares its exponent.  Otherwise (about 2^-19 of the
// products, or any zero, subnormal or overflowing one) the integer
// evaluation decides, so the warp almost never takes that path.
__device__ __forceinline__ unsigned term_exponent_fast(float c, float r, float a) {
  const float cr = fabsf(c * r);
  const float p = cr * fabsf(a);
  const unsigned bcr = __float_as_uint(cr), bp = __float_as_uint(p);
  const unsigned ecr = bcr >> 23, ex = bp >> 23, m = bp & 0x7FFFFFu;
  if (ecr != 0 && ecr < 255 && ex != 0 && ex < 255 && m >= 8u && m <= 0x7FFFF7u)
    return ex - 126u + static_cast<unsigned>(kEBias);
  return term_exponent(c, r, a);
}

// Candidate i of an Algorithm 1 grid, fl32(x0 + i * step) in float64.
__device__ __forceinline__ float cand_at(double x0, double step, int i) {
  return static_cast<float>(x0 + static_cast<double>(i) * step);
}

// First candidate index i with r <= cand[i] (strict=false) or r < cand[i]
// (strict=true); n if none.  Candidates ascend.
__device__ __forceinline__ int first_cand(const float* cand, int n, float r, bool strict) {
  int lo = 0, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    const float c = cand[mid];
    const bool ok = strict ? (r < c) : (r <= c);
    if (ok) hi = mid; else lo = mid + 1;
  }
  return lo;
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// ------------------------------------------------------------------ passes
// Scalar results a thread accumulates over its tokens.
struct PassAcc {
  unsigned long long n_neg, n_pos, k_bf, k_fp;
  long long s_pos_bf, s_neg_bf, s_neg_fp, s_pos_fp;
  unsigned emax, bad, nb_below1, nb_above, nb_m, nb_M1;
  unsigned l_below, l_in;  // per-thread counts: T / grid threads each at most
  long long h_below;
  unsigned l_nb_below1, l_nb_above_inv, l_mp_inv, l_Mp1;
  unsigned h_nb_below1, h_nb_above_inv, h_top1, h_mp_inv, h_Mp1;
  unsigned long long n_valid;  // last: zero from the initialiser's omitted tail
};

// Constants of one pass.
struct PassCtx {
  int stage, digit, shift;
  bool grid_mode;
  float lo_star, hi_star;
  unsigned prefix, u, key_lm, key_lM, key_hm, key_hM;
};

// One token of a pass: updates the thread's scalars and returns the
// histogram bin the token adds `w` to (-1: none).
template <int STAGE>
__device__ __forceinline__ int pass_token(const Args& a, const PassCtx& x, const float* sh_cand,
                                          bool valid, float A, float rf, float rb, float c,
                                          PassAcc& acc, long long& w, unsigned& cand) {
  w = 0;
  cand = kNone;  // the token's key when it goes to a list
  const bool neg = valid && A < 0.f, pos = valid && A > 0.f;
  if (STAGE == kPrep) {
    if (!(isfinite(A) && isfinite(rf) && isfinite(rb) && isfinite(c)) || rf < 0.f || rb < 0.f ||
        c < 0.f)
      acc.bad = 1;
    acc.n_valid += valid;
    if (neg) {
      ++acc.n_neg;
      if (rb <= a.c_lo) ++acc.k_bf;
    }
    if (pos) ++acc.n_pos;
    if (neg || pos) {
      // |fl64(fl64(c r) A)| is non-decreasing in r (c r is exact, the rounding
      // monotone), so the larger ratio gives the larger of the two exponents
      acc.emax = max(acc.emax, term_exponent_fast(c, fmaxf(rb, rf), A));
    }
    if (!neg) return -1;
    w = 1;
    if (x.grid_mode) return first_cand(sh_cand, a.n_lcand, rf, false);
    const unsigned key = key_of(rf);
    if (key < x.key_lm) {
      ++acc.l_below;
      acc.l_nb_below1 = max(acc.l_nb_below1, key + 1);
      return -1;
    }
    if (key > x.key_lM) {
      acc.l_nb_above_inv = max(acc.l_nb_above_inv, ~key);
      return -1;
    }
    ++acc.l_in;
    if (key > x.key_lm) acc.l_mp_inv = max(acc.l_mp_inv, ~key);
    acc.l_Mp1 = max(acc.l_Mp1, key + 1);
    cand = key;
    return static_cast<int>(digit_of(key, 0));
  }
  if (STAGE == kSums) {
    if (!(neg || pos)) return -1;
    const long long qb = fixed_term(c, rb, A, x.shift);
    if (pos && rb < a.c_hi) acc.s_pos_bf += qb;
    if (neg && rb > a.c_lo) acc.s_neg_bf += qb;
    if (x.grid_mode) {
      const long long qf = fixed_term(c, rf, A, x.shift);
      if (neg && rf > x.lo_star) acc.s_neg_fp += qf;
      if (neg && rf <= x.lo_star) ++acc.k_fp;
      if (!pos) return -1;
      w = qf;
      return first_cand(sh_cand, a.n_hcand, rf, true);
    }
    if (!neg) return -1;
    const unsigned key = key_of(rf);
    if (key < x.key_lm || key > x.key_lM || !digit_match(key, 1, x.prefix)) return -1;
    w = 1;
    return static_cast<int>(digit_of(key, 1));
  }
  // H stages: Pos set, weights q_fp8.  kH0 needs q_fp8 for both signs: one
  // evaluation for every signed token keeps the warp on one path.
  if (STAGE == kH0) {
    if (!(neg || pos)) return -1;
    const long long qf = fixed_term(c, rf, A, x.shift);
    if (neg) {
      if (rf > x.lo_star) acc.s_neg_fp += qf;
      else ++acc.k_fp;
      return -1;
    }
    const unsigned key = key_of(rf);
    if (key < x.key_hm) {
      acc.h_below += qf;
      if (qf != 0) acc.h_nb_below1 = max(acc.h_nb_below1, key + 1);
      return -1;
    }
    if (key >= x.key_hM) {
      if (qf != 0) {
        acc.h_nb_above_inv = max(acc.h_nb_above_inv, ~key);
        acc.h_top1 = max(acc.h_top1, key + 1);
      }
      return -1;
    }
    if (qf != 0) {
      acc.h_mp_inv = max(acc.h_mp_inv, ~key);
      acc.h_Mp1 = max(acc.h_Mp1, key + 1);
    }
    cand = key;
    w = qf;
    return static_cast<int>(digit_of(key, 0));
  }
  // GRID mode's P(H*) pass (EXACT mode takes P(H*) from the I_H list)
  if (!pos) return -1;
  if (STAGE == kPFin) {
    if (rf < x.hi_star) acc.s_pos_fp += fixed_term(c, rf, A, x.shift);
    return -1;
  }
  return -1;
}

// Block histogram in shared memory with native 32-bit atomics only: counts
// as 32-bit words, 64-bit weights as low and high words, the carry out of the
// low word taken from the value the atomic returns (exact modulo 2^64).
struct __align__(16) ShHist {
  unsigned cnt[kBuckets];
  unsigned wlo[kBuckets];
  unsigned whi[kBuckets];
};

__device__ __forceinline__ void sh_add(ShHist& h, int d, unsigned n, unsigned long long w) {
  atomicAdd(&h.cnt[d], n);
  const unsigned lo = static_cast<unsigned>(w), hi = static_cast<unsigned>(w >> 32);
  const unsigned old = lo ? atomicAdd(&h.wlo[d], lo) : 0u;
  const unsigned carry = (old + lo < old) ? 1u : 0u;
  if (hi + carry) atomicAdd(&h.whi[d], hi + carry);
}

// Adds every lane's (bin d, weight w >= 0) to the block histogram with one
// update per distinct bin of the warp: ratios crowd into few bins of a
// leading digit.  Weights are summed in three 21-bit slices by 32-bit warp
// reductions (32 slices cannot overflow).  Called by all 32 lanes together;
// d < 0 adds nothing.
template <bool COUNTS>
__device__ __forceinline__ void hist_add_warp(ShHist& sh, int d, long long w) {
  const int lane = threadIdx.x & 31;
  unsigned pending = __ballot_sync(0xffffffffu, d >= 0);
  while (pending) {
    const int leader = __ffs(pending) - 1;
    const int dl = __shfl_sync(0xffffffffu, d, leader);
    const bool mine = d == dl;
    const unsigned grp = __ballot_sync(0xffffffffu, mine);
    unsigned long long sum = __popc(grp);
    if (!COUNTS) {
      const unsigned long long v = mine ? static_cast<unsigned long long>(w) : 0ull;
      const unsigned s0 = __reduce_add_sync(0xffffffffu, static_cast<unsigned>(v & 0x1FFFFFu));
      const unsigned s1 = __reduce_add_sync(0xffffffffu, static_cast<unsigned>((v >> 21) & 0x1FFFFFu));
      const unsigned s2 = __reduce_add_sync(0xffffffffu, static_cast<unsigned>(v >> 42));
      sum = static_cast<unsigned long long>(s0) + (static_cast<unsigned long long>(s1) << 21) +
            (static_cast<unsigned long long>(s2) << 42);
    }
    if (lane == leader) sh_add(sh, dl, __popc(grp), sum);
    pending &= ~grp;
  }
}

// Per-lane update, for digits whose bins are spread out.
__device__ __forceinline__ void hist_add_lane(ShHist& sh, int d, long long w) {
  if (d >= 0) sh_add(sh, d, 1u, static_cast<unsigned long long>(w));
}

// One pass over the tokens by the whole grid (or by one block in the fused
// small-T kernel).  Passes read G tokens per lane and step: 16-byte loads when
// G = 4.  sh_cand holds the stage's grid candidates in GRID mode.
template <int G, int STAGE>
__device__ void pass_body(const Args& a, ShHist& sh, float* sh_cand) {
  // full passes over the tokens: kPrep, kSums, kH0 and GRID mode's kPFin
  constexpr int stage = STAGE;
  State* st = a.st;
  if (stage == kPFin && st->p_known) return;
  const bool grid_mode = a.grid_mode != 0;
  const bool want_hist = grid_mode ? (stage == kPrep || stage == kSums)
                                   : (stage == kPrep || stage == kSums || stage == kH0);
  if (want_hist) {
    for (int i = threadIdx.x; i < kBuckets; i += blockDim.x) {
      sh.cnt[i] = 0;
      sh.wlo[i] = 0;
      sh.whi[i] = 0;
      if (grid_mode) {
        const bool lower = stage == kPrep;
        const int n = lower ? a.n_lcand : a.n_hcand;
        sh_cand[i] = i < n ? cand_at(lower ? a.lo_grid0 : a.hi_grid0, a.step, i) : 0.f;
      }
    }
    __syncthreads();
  }
  const int shift = st->shift;
  const float lo_star = st->lo_star, hi_star = st->hi_star;
  const unsigned prefix = st->prefix, u = st->u_key;
  const int digit = stage == kSums ? 1 : 0;
  const unsigned key_lm = key_of(a.lo_min), key_lM = key_of(a.lo_max);
  const unsigned key_hm = key_of(a.hi_min), key_hM = key_of(a.hi_max);

  PassCtx x;
  x.stage = stage;
  x.digit = digit;
  x.shift = shift;
  x.grid_mode = grid_mode;
  x.lo_star = lo_star;
  x.hi_star = hi_star;
  x.prefix = prefix;
  x.u = u;
  x.key_lm = key_lm;
  x.key_lM = key_lM;
  x.key_hm = key_hm;
  x.key_hM = key_hM;
  PassAcc acc{0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, kNone, kNone, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0};
  // EXACT mode writes the tokens inside the interval to its list: I_L from
  // the first pass, I_H (with q_fp8) from the H digit-0 pass, each warp into
  // its own segment
  const bool to_list = !grid_mode && (stage == kPrep || stage == kH0);
  const unsigned seg = static_cast<unsigned>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const size_t seg0 = static_cast<size_t>(seg) * a.seg_cap;
  unsigned* list_keys = stage == kPrep ? a.l_keys : a.h_keys;
  unsigned seg_fill = 0;
  // histogram update: 0 none, 1 warp-aggregated counts, 2 warp-aggregated
  // weights (leading digit, grid candidates), 3 per lane (later digits)
  int hist_mode = 0;
  if (want_hist) {
    if (stage == kPrep) hist_mode = 1;
    else if (stage == kH0 || (grid_mode && stage == kSums)) hist_mode = 2;
    else hist_mode = 3;
  }
  const bool need_rb = stage == kPrep || stage == kSums;
  const bool need_c = a.coef != nullptr;
  const int lane = threadIdx.x & 31;
  // append to the warp's segment (warp-uniform fill)
  auto append = [&](unsigned cand, long long q) {
    const unsigned want = __ballot_sync(0xffffffffu, cand != kNone);
    if (!want) return;
    if (cand != kNone) {
      const size_t i = seg0 + seg_fill + __popc(want & ((1u << lane) - 1u));
      list_keys[i] = cand;
      if (stage == kH0) a.h_q[i] = q;
    }
    seg_fill += __popc(want);
  };
  const int64_t ng = a.T / G;
  const int64_t warp_id = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  // warp-uniform steps: every lane runs every step (the histogram update is
  // a warp collective); lanes past the end see invalid zero tokens
  for (int64_t base = warp_id * 32; base < ng; base += nwarps * 32) {
    const int64_t g = base + lane;
    const bool in = g < ng;
    float rf[G], A[G], rb[G], c[G];
    bool valid[G];
#pragma unroll
    for (int j = 0; j < G; ++j) {
      rf[j] = 0.f;
      A[j] = 0.f;
      rb[j] = 0.f;
      c[j] = 1.f;
      valid[j] = false;
    }
    if (in) {
      if (G == 4) {
        const float4 vf = __ldg(reinterpret_cast<const float4*>(a.r_fp8) + g);
        const float4 va = __ldg(reinterpret_cast<const float4*>(a.adv) + g);
        rf[0] = vf.x; rf[1] = vf.y; rf[2] = vf.z; rf[3] = vf.w;
        A[0] = va.x; A[1] = va.y; A[2] = va.z; A[3] = va.w;
        if (need_rb) {
          const float4 vb = __ldg(reinterpret_cast<const float4*>(a.r_bf16) + g);
          rb[0] = vb.x; rb[1] = vb.y; rb[2] = vb.z; rb[3] = vb.w;
        }
        if (need_c) {
          const float4 vc = __ldg(reinterpret_cast<const float4*>(a.coef) + g);
          c[0] = vc.x; c[1] = vc.y; c[2] = vc.z; c[3] = vc.w;
        }
        const uint32_t m = a.mask ? __ldg(reinterpret_cast<const uint32_t*>(a.mask) + g) : 0x01010101u;
#pragma unroll
        for (int j = 0; j < G; ++j) valid[j] = ((m >> (8 * j)) & 0xFFu) != 0;
      } else {
        rf[0] = a.r_fp8[g];
        A[0] = a.adv[g];
        if (need_rb) rb[0] = a.r_bf16[g];
        if (need_c) c[0] = a.coef[g];
        valid[0] = a.mask ? a.mask[g] != 0 : true;
      }
    }
#pragma unroll
    for (int j = 0; j < G; ++j) {
      long long w;
      unsigned cand;
      const int d = pass_token<STAGE>(a, x, sh_cand, valid[j], A[j], rf[j], rb[j], c[j], acc, w, cand);
      if (to_list) append(cand, w);
      if (hist_mode == 1) hist_add_warp<true>(sh, d, w);
      else if (hist_mode == 2) hist_add_warp<false>(sh, d, w);
      else if (hist_mode == 3) hist_add_lane(sh, d, w);
    }
  }
  if (G > 1 && blockIdx.x == 0 && threadIdx.x < 32) {  // the last T mod 4 tokens
    const int64_t t = ng * G + lane;
    const bool in = t < a.T;
    const float rf = in ? a.r_fp8[t] : 0.f;
    const float A = in ? a.adv[t] : 0.f;
    const float rb = in && need_rb ? a.r_bf16[t] : 0.f;
    const float c = in && need_c ? a.coef[t] : 1.f;
    const bool valid = in && (a.mask ? a.mask[t] != 0 : true);
    long long w;
    unsigned cand;
    const int d = pass_token<STAGE>(a, x, sh_cand, valid, A, rf, rb, c, acc, w, cand);
    if (to_list) append(cand, w);
    if (hist_mode == 1) hist_add_warp<true>(sh, d, w);
    else if (hist_mode == 2) hist_add_warp<false>(sh, d, w);
    else if (hist_mode == 3) hist_add_lane(sh, d, w);
  }
  if (to_list && lane == 0) (stage == kPrep ? a.l_cnt : a.h_cnt)[seg] = seg_fill;
  unsigned long long n_neg = acc.n_neg, n_pos = acc.n_pos, k_bf = acc.k_bf, k_fp = acc.k_fp,
                     n_valid = acc.n_valid;
  long long s_pos_bf = acc.s_pos_bf, s_neg_bf = acc.s_neg_bf, s_neg_fp = acc.s_neg_fp,
            s_pos_fp = acc.s_pos_fp;
  unsigned emax = acc.emax, bad = acc.bad;
  unsigned nb_below1 = acc.nb_below1, nb_above = acc.nb_above, nb_m = acc.nb_m, nb_M1 = acc.nb_M1;
  unsigned long long l_below = acc.l_below, l_in = acc.l_in;  // widened for the warp sum
  long long h_below = acc.h_below;

  // ---- flush: warp-aggregated scalars, then the block histogram
  n_neg = warp_sum(n_neg);
  n_pos = warp_sum(n_pos);
  n_valid = warp_sum(n_valid);
  k_bf = warp_sum(k_bf);
  k_fp = warp_sum(k_fp);
  s_pos_bf = warp_sum(s_pos_bf);
  s_neg_bf = warp_sum(s_neg_bf);
  s_neg_fp = warp_sum(s_neg_fp);
  s_pos_fp = warp_sum(s_pos_fp);
  emax = __reduce_max_sync(0xffffffffu, emax);
  bad = __reduce_or_sync(0xffffffffu, bad);
  nb_below1 = __reduce_max_sync(0xffffffffu, nb_below1);
  nb_above = __reduce_min_sync(0xffffffffu, nb_above);
  nb_m = __reduce_min_sync(0xffffffffu, nb_m);
  nb_M1 = __reduce_max_sync(0xffffffffu, nb_M1);
  l_below = warp_sum(l_below);
  l_in = warp_sum(l_in);
  h_below = warp_sum(h_below);
  unsigned ext[9] = {acc.l_nb_below1, acc.l_nb_above_inv, acc.l_mp_inv, acc.l_Mp1, acc.h_nb_below1,
                     acc.h_nb_above_inv, acc.h_top1, acc.h_mp_inv, acc.h_Mp1};
  unsigned* ext_st[9] = {&st->l_nb_below1, &st->l_nb_above_inv, &st->l_mp_inv, &st->l_Mp1, &st->h_nb_below1,
                         &st->h_nb_above_inv, &st->h_top1, &st->h_mp_inv, &st->h_Mp1};
#pragma unroll
  for (int i = 0; i < 9; ++i) ext[i] = __reduce_max_sync(0xffffffffu, ext[i]);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < 9; ++i)
      if (ext[i]) atomicMax(ext_st[i], ext[i]);
    if (l_below) atomicAdd(&st->l_below, l_below);
    if (l_in) atomicAdd(&st->l_in, l_in);
    if (h_below) atomicAdd(&st->h_below, static_cast<unsigned long long>(h_below));
    if (n_neg) atomicAdd(&st->n_neg, n_neg);
    if (n_pos) atomicAdd(&st->n_pos, n_pos);
    if (n_valid) atomicAdd(&st->n_valid, n_valid);
    if (k_bf) atomicAdd(&st->k_bf16, k_bf);
    if (k_fp) atomicAdd(&st->k_fp8, k_fp);
    if (s_pos_bf) atomicAdd(&st->s_pos_bf, static_cast<unsigned long long>(s_pos_bf));
    if (s_neg_bf) atomicAdd(&st->s_neg_bf, static_cast<unsigned long long>(s_neg_bf));
    if (s_neg_fp) atomicAdd(&st->s_neg_fp, static_cast<unsigned long long>(s_neg_fp));
    if (s_pos_fp) atomicAdd(&st->s_pos_fp, static_cast<unsigned long long>(s_pos_fp));
    if (emax) atomicMax(&st->emax_bits, static_cast<unsigned long long>(emax));
    if (bad) {
      atomicOr(&st->bad, 1u);
      flag(kErrDevice);
    }
    if (nb_below1) atomicMax(&st->nb_below1, nb_below1);
    if (nb_above != kNone) atomicMin(&st->nb_above, nb_above);
    if (nb_m != kNone) atomicMin(&st->nb_mpiece, nb_m);
    if (nb_M1) atomicMax(&st->nb_Mpiece1, nb_M1);
  }
  if (want_hist) {
    __syncthreads();
    for (int i = threadIdx.x; i < kBuckets; i += blockDim.x) {
      if (sh.cnt[i]) {
        atomicAdd(&st->h_cnt[i], static_cast<unsigned long long>(sh.cnt[i]));
        atomicAdd(&st->h_w[i], (static_cast<unsigned long long>(sh.whi[i]) << 32) | sh.wlo[i]);
      }
    }
  }
}

// EXACT mode's later selection passes read the interval lists only:
//   kL2   L digit 2 of the I_L keys (counts)
//   kLNb  the I_L keys next to u (the ones outside I_L were kept by kPrep)
//   kH1, kH2  H digits 1 and 2 of the I_H keys, weighted by q_fp8
//   kHNb  the q != 0 keys of I_H next to u
//   kPFin P(H*) = P(hi_min) + the q of I_H keys below H*
template <int STAGE>
__device__ void list_body(const Args& a, ShHist& sh) {
  State* st = a.st;
  if ((STAGE == kH1 || STAGE == kH2 || STAGE == kHNb) && !st->h_active) return;
  if (STAGE == kPFin && st->p_known) return;
  constexpr bool lower = STAGE == kL2 || STAGE == kLNb;
  constexpr bool want_hist = STAGE == kL2 || STAGE == kH1 || STAGE == kH2;
  constexpr int digit = STAGE == kH1 ? 1 : 2;
  if (want_hist) {
    for (int i = threadIdx.x; i < kBuckets; i += blockDim.x) {
      sh.cnt[i] = 0;
      sh.wlo[i] = 0;
      sh.whi[i] = 0;
    }
    __syncthreads();
  }
  const unsigned prefix = st->prefix, u = st->u_key, key_h = key_of(st->hi_star);
  const unsigned* cnt = lower ? a.l_cnt : a.h_cnt;
  const int lane = threadIdx.x & 31;
  const unsigned nwarps = (gridDim.x * blockDim.x) >> 5;
  unsigned nb_below1 = 0, nb_above = kNone;
  long long p = 0;
  for (unsigned sg = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; sg < a.nseg; sg += nwarps) {
    const unsigned fill = cnt[sg];
    for (unsigned j = lane; j < fill; j += 32) {
      const size_t i = static_cast<size_t>(sg) * a.seg_cap + j;
      const unsigned key = lower ? a.l_keys[i] : a.h_keys[i];
      if (STAGE == kL2) {
        if (digit_match(key, 2, prefix)) hist_add_lane(sh, static_cast<int>(digit_of(key, 2)), 1);
      } else if (STAGE == kLNb) {
        if (key < u) nb_below1 = max(nb_below1, key + 1);
        if (key > u) nb_above = min(nb_above, key);
      } else {
        const long long q = a.h_q[i];
        if (STAGE == kH1 || STAGE == kH2) {
          if (digit_match(key, digit, prefix)) hist_add_lane(sh, static_cast<int>(digit_of(key, digit)), q);
        } else if (STAGE == kHNb) {
          if (q != 0) {
            if (key < u) nb_below1 = max(nb_below1, key + 1);
            if (key > u) nb_above = min(nb_above, key);
          }
        } else if (key < key_h) {  // kPFin: r < H*
          p += q;
        }
      }
    }
  }
  if (STAGE == kPFin && blockIdx.x == 0 && threadIdx.x == 0) p += static_cast<long long>(st->h_below);
  nb_below1 = __reduce_max_sync(0xffffffffu, nb_below1);
  nb_above = __reduce_min_sync(0xffffffffu, nb_above);
  p = warp_sum(p);
  if (lane == 0) {
    if (nb_below1) atomicMax(&st->nb_below1, nb_below1);
    if (nb_above != kNone) atomicMin(&st->nb_above, nb_above);
    if (p) atomicAdd(&st->s_pos_fp, static_cast<unsigned long long>(p));
  }
  if (want_hist) {
    __syncthreads();
    for (int i = threadIdx.x; i < kBuckets; i += blockDim.x) {
      if (sh.cnt[i]) {
        atomicAdd(&st->h_cnt[i], static_cast<unsigned long long>(sh.cnt[i]));
        atomicAdd(&st->h_w[i], (static_cast<unsigned long long>(sh.whi[i]) << 32) | sh.wlo[i]);
      }
    }
  }
}

// One pass, compiled per stage so that each holds only its own state.
template <int G>
__device__ void pass_any(const Args& a, int stage, ShHist& sh, float* sh_cand) {
  switch (stage) {
    case kPrep: pass_body<G, kPrep>(a, sh, sh_cand); break;
    case kSums: pass_body<G, kSums>(a, sh, sh_cand); break;
    case kL2: list_body<kL2>(a, sh); break;
    case kLNb: list_body<kLNb>(a, sh); break;
    case kH0: pass_body<G, kH0>(a, sh, sh_cand); break;
    case kH1: list_body<kH1>(a, sh); break;
    case kH2: list_body<kH2>(a, sh); break;
    case kHNb: list_body<kHNb>(a, sh); break;
    default:
      if (a.grid_mode) pass_body<G, kPFin>(a, sh, sh_cand);
      else list_body<kPFin>(a, sh);
      break;
  }
}

template <int G, int STAGE>
__global__ void __launch_bounds__(256) pass_kernel(Args a) {
  __shared__ ShHist sh;
  __shared__ float sh_cand[kBuckets];
  pass_body<G, STAGE>(a, sh, sh_cand);
}

template <int STAGE>
__global__ void __launch_bounds__(256) list_kernel(Args a) {
  __shared__ ShHist sh;
  list_body<STAGE>(a, sh);
}

template <int G>
void launch_pass(const Args& a, int stage, int grid, cudaStream_t s) {
  switch (stage) {
    case kPrep: pass_kernel<G, kPrep><<<grid, 256, 0, s>>>(a); break;
    case kSums: pass_kernel<G, kSums><<<grid, 256, 0, s>>>(a); break;
    case kL2: list_kernel<kL2><<<grid, 256, 0, s>>>(a); break;
    case kLNb: list_kernel<kLNb><<<grid, 256, 0, s>>>(a); break;
    case kH0: pass_kernel<G, kH0><<<grid, 256, 0, s>>>(a); break;
    case kH1: list_kernel<kH1><<<grid, 256, 0, s>>>(a); break;
    case kH2: list_kernel<kH2><<<grid, 256, 0, s>>>(a); break;
    case kHNb: list_kernel<kHNb><<<grid, 256, 0, s>>>(a); break;
    default:
      if (a.grid_mode) pass_kernel<G, kPFin><<<grid, 256, 0, s>>>(a);
      else list_kernel<kPFin><<<grid, 256, 0, s>>>(a);
      break;
  }
}

// ------------------------------------------------------------------ 128-bit
struct U128 {
  unsigned long long hi, lo;
};
__device__ __forceinline__ U128 mul_u64(unsigned long long a, unsigned long long b) {
  return U128{__umul64hi(a, b), a * b};
}
__device__ __forceinline__ bool ge128(U128 a, U128 b) {
  return a.hi > b.hi || (a.hi == b.hi && a.lo >= b.lo);
}
__device__ __forceinline__ bool lt128(U128 a, U128 b) { return !ge128(a, b); }
__device__ __forceinline__ U128 sub128(U128 a, U128 b) {  // a >= b
  U128 r;
  r.lo = a.lo - b.lo;
  r.hi = a.hi - b.hi - (a.lo < b.lo ? 1ull : 0ull);
  return r;
}
__device__ __forceinline__ U128 absdiff128(U128 a, U128 b) { return ge128(a, b) ? sub128(a, b) : sub128(b, a); }

__device__ __forceinline__ float next_up(float x) { return nextafterf(x, INFINITY); }
__device__ __forceinline__ float next_down(float x) { return nextafterf(x, -INFINITY); }
__device__ __forceinline__ float clampf(float x, float lo, float hi) { return fminf(fmaxf(x, lo), hi); }

__device__ __forceinline__ float smooth(float b_old, float b_star, float delta) {
  if (isnan(b_old)) return b_star;
  float d = __fmul_rn(__fsub_rn(b_star, b_old), 0.5f);
  d = fminf(fmaxf(d, -delta), delta);
  return __fadd_rn(b_old, d);
}

// One step of the weighted radix select, by the whole block (512 or 1024
// threads): smallest bucket b with cnt[b] > 0 and
// (below + sum_{b' <= b} w[b']) * D >= X.  sh_incl: kBuckets of shared scratch.
__device__ void select_step(State* st, int bits, bool last, long long* sh_incl) {
  __shared__ long long warp_tot[32];
  __shared__ int sh_best;
  const int nb = 1 << bits;
  const int tid = threadIdx.x;
  const int per = kBuckets / blockDim.x;  // 2 or 4 buckets per thread
  long long local[4] = {0, 0, 0, 0};
  long long run = 0;
  for (int j = 0; j < per; ++j) {
    const int b = tid * per + j;
    run += (b < nb) ? static_cast<long long>(st->h_w[b]) : 0;
    local[j] = run;
  }
  // exclusive scan of per-thread totals
  const int lane = tid & 31, wid = tid >> 5;
  long long v = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  if (lane == 31) warp_tot[wid] = v;
  if (tid == 0) sh_best = 0x7FFFFFFF;
  __syncthreads();
  if (wid == 0) {
    long long w = (lane < (int)(blockDim.x >> 5)) ? warp_tot[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long n = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += n;
    }
    warp_tot[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  const long long before = (v - run) + (wid > 0 ? warp_tot[wid - 1] : 0);
  const U128 X{st->tgt_hi, st->tgt_lo};
  const unsigned long long D = static_cast<unsigned long long>(st->dmul);
  for (int j = 0; j < per; ++j) {
    const int b = tid * per + j;
    const long long incl = before + local[j];
    sh_incl[b] = incl;
    if (b < nb && st->h_cnt[b] > 0) {
      const long long cum = st->below + incl;
      if (ge128(mul_u64(static_cast<unsigned long long>(cum), D), X)) atomicMin(&sh_best, b);
    }
  }
  __syncthreads();
  if (tid == 0) {
    const int b = sh_best;
    if (b == 0x7FFFFFFF) {
      st->found = 0;
    } else {
      const long long excl = sh_incl[b] - static_cast<long long>(st->h_w[b]);
      st->below += excl;
      st->prefix = (st->prefix << bits) | static_cast<unsigned>(b);
      if (last) {
        st->u_key = st->prefix;
        st->p_lt = st->below;
        st->p_le = st->below + static_cast<long long>(st->h_w[b]);
      }
    }
  }
  __syncthreads();
  for (int i = tid; i < kBuckets; i += blockDim.x) {
    st->h_cnt[i] = 0;
    st->h_w[i] = 0;
  }
}

__device__ void reset_neighbours(State* st) {
  st->nb_below1 = 0;
  st->nb_above = kNone;
  st->nb_mpiece = kNone;
  st->nb_Mpiece1 = 0;
}

// Decides stage 2's target after D_fp8 is known; false when degenerate (H* is
// then the reference bound clamped to I_H).
__device__ bool begin_upper(const Args& a, State* st) {
  const long long n_bf = static_cast<long long>(st->s_pos_bf);
  const long long d_bf = llabs(static_cast<long long>(st->s_neg_bf));
  const long long d_fp = llabs(static_cast<long long>(st->s_neg_fp));
  int fl = st->flags;
  if (st->n_pos == 0) fl |= FP8RL_CALIB_FLAG_NO_POS;
  if (d_bf == 0) fl |= FP8RL_CALIB_FLAG_ZERO_D_BF16;
  if (d_fp == 0) fl |= FP8RL_CALIB_FLAG_ZERO_D_FP8;
  st->flags = fl;
  const U128 X = mul_u64(static_cast<unsigned long long>(n_bf), static_cast<unsigned long long>(d_fp));
  st->tgt_hi = X.hi;
  st->tgt_lo = X.lo;
  st->dmul = d_bf;
  st->below = 0;
  st->prefix = 0;
  st->found = 1;
  const bool active =
      !(fl & (FP8RL_CALIB_FLAG_NO_POS | FP8RL_CALIB_FLAG_ZERO_D_BF16 | FP8RL_CALIB_FLAG_ZERO_D_FP8));
  st->h_active = active;
  if (!active) st->hi_star = clampf(a.c_hi, a.hi_min, a.hi_max);
  return active;
}

__device__ void write_result(const Args& a, State* st) {
  fp8rl_calib_result r;
  r.lo_star = st->lo_star;
  r.hi_star = st->hi_star;
  r.lo_new = smooth(a.lo_old, st->lo_star, a.delta_lo);
  r.hi_new = smooth(a.hi_old, st->hi_star, a.delta_hi);
  r.c_lo = a.c_lo;
  r.c_hi = a.c_hi;
  r.flags = st->flags;
  r.shift = st->shift;
  r.n_neg = static_cast<int64_t>(st->n_neg);
  r.n_pos = static_cast<int64_t>(st->n_pos);
  r.k_bf16 = static_cast<int64_t>(st->k_bf16);
  r.k_fp8 = static_cast<int64_t>(st->k_fp8);
  r.sum_pos_bf16 = static_cast<int64_t>(st->s_pos_bf);
  r.sum_neg_bf16 = llabs(static_cast<long long>(st->s_neg_bf));
  r.sum_neg_fp8 = llabs(static_cast<long long>(st->s_neg_fp));
  r.sum_pos_fp8 = static_cast<int64_t>(st->s_pos_fp);
  r.rho_bf16 = r.sum_neg_bf16 ? static_cast<double>(r.sum_pos_bf16) / static_cast<double>(r.sum_neg_bf16) : NAN;
  r.rho_fp8 = r.sum_neg_fp8 ? static_cast<double>(r.sum_pos_fp8) / static_cast<double>(r.sum_neg_fp8) : NAN;
  r.n_valid = static_cast<int64_t>(st->n_valid);
  *a.out = r;
}

__device__ void zero_hist(State* st) {
  for (int i = threadIdx.x; i < kBuckets; i += blockDim.x) {
    st->h_cnt[i] = 0;
    st->h_w[i] = 0;
  }
}

// L* from the unconstrained minimiser interval [lo, hi] of |C(L) - k| (closed
// in float32) and the pieces of C containing the ends of I_L.
__device__ float lower_from_interval(const Args& a, const State* st, float lo, float hi) {
  if (fmaxf(lo, a.lo_min) <= fminf(hi, a.lo_max))
    return clampf(a.c_lo, fmaxf(lo, a.lo_min), fminf(hi, a.lo_max));
  if (hi < a.lo_min) {  // f increases across I_L: the piece containing lo_min
    const float b = st->nb_mpiece != kNone ? next_down(__uint_as_float(st->nb_mpiece)) : INFINITY;
    return clampf(a.c_lo, a.lo_min, fminf(b, a.lo_max));
  }
  // f decreases across I_L: the piece containing lo_max
  const float b = st->nb_Mpiece1 ? __uint_as_float(st->nb_Mpiece1 - 1) : -INFINITY;
  return clampf(a.c_lo, fmaxf(b, a.lo_min), a.lo_max);
}

__device__ float upper_from_interval(const Args& a, const State* st, float lo, float hi) {
  if (fmaxf(lo, a.hi_min) <= fminf(hi, a.hi_max))
    return clampf(a.c_hi, fmaxf(lo, a.hi_min), fminf(hi, a.hi_max));
  if (hi < a.hi_min) {  // the piece (z, b] containing hi_min
    const float b = st->nb_mpiece != kNone ? __uint_as_float(st->nb_mpiece) : INFINITY;
    return clampf(a.c_hi, a.hi_min, fminf(b, a.hi_max));
  }
  // the piece containing hi_max
  const float b = st->nb_Mpiece1 ? next_up(__uint_as_float(st->nb_Mpiece1 - 1)) : -INFINITY;
  return clampf(a.c_hi, fmaxf(b, a.hi_min), a.hi_max);
}

__device__ void decide_body(const Args& a, int stage, long long* scratch) {
  State* st = a.st;
  const int tid = threadIdx.x;
  __shared__ int sh_go;

  if (stage == kPrep) {
    if (tid == 0) {
      // fixed-point shift s = 62 - E - B: max|e| < 2^E, 2^B >= signed tokens
      const unsigned long long nt = st->n_neg + st->n_pos;
      int s = 0;
      if (nt > 0 && st->emax_bits > 0) {
        const int E = static_cast<int>(st->emax_bits) - kEBias;
        const int B = nt > 1 ? 64 - __clzll(static_cast<long long>(nt - 1)) : 0;
        s = 62 - E - B;
      }
      st->shift = s;
      st->flags = 0;
      if (st->n_neg == 0) {
        st->flags |= FP8RL_CALIB_FLAG_NO_NEG;
        st->lo_star = clampf(a.c_lo, a.lo_min, a.lo_max);
      }
      st->tgt_hi = 0;
      st->tgt_lo = st->k_bf16;
      st->dmul = 1;
      st->below = static_cast<long long>(st->l_below);  // A<0 tokens under I_L (0 in GRID mode)
      st->prefix = 0;
      st->found = 1;
      sh_go = st->n_neg > 0;
      if (a.grid_mode && st->n_neg > 0) {
        // cnt_le(L_i) is the prefix sum of the candidate histogram; minimise
        // (|cnt - k|, |L_i - c_lo|, L_i) over the <= 2047 candidates
        const long long k = static_cast<long long>(st->k_bf16);
        long long cum = 0, best_f = -1;
        double best_d = 0;
        float best = 0;
        for (int i = 0; i < a.n_lcand; ++i) {
          cum += static_cast<long long>(st->h_cnt[i]);
          const long long f = llabs(cum - k);
          const float L = cand_at(a.lo_grid0, a.step, i);
          const double d = fabs(static_cast<double>(L) - static_cast<double>(a.c_lo));
          if (best_f < 0 || f < best_f || (f == best_f && (d < best_d || (d == best_d && L < best)))) {
            best_f = f;
            best_d = d;
            best = L;
          }
        }
        st->lo_star = best;
      }
    }
    __syncthreads();
    if (a.grid_mode) zero_hist(st);
    else if (sh_go) select_step(st, 11, false, scratch);
    return;
  }

  if (stage == kSums) {
    if (!a.grid_mode) {
      if (st->n_neg > 0) select_step(st, 11, false, scratch);
      return;
    }
    if (tid == 0 && begin_upper(a, st)) {
      const U128 X{st->tgt_hi, st->tgt_lo};
      const unsigned long long D = static_cast<unsigned long long>(st->dmul);
      long long cum = 0;
      U128 best_f{0, 0};
      double best_d = 0;
      float best = 0;
      bool have = false;
      for (int j = 0; j < a.n_hcand; ++j) {
        cum += static_cast<long long>(st->h_w[j]);
        const U128 f = absdiff128(mul_u64(static_cast<unsigned long long>(cum), D), X);
        const float H = cand_at(a.hi_grid0, a.step, j);
        const double d = fabs(static_cast<double>(H) - static_cast<double>(a.c_hi));
        const bool better = !have || lt128(f, best_f) ||
                            (!lt128(best_f, f) && (d < best_d || (d == best_d && H < best)));
        if (better) {
          best_f = f;
          best_d = d;
          best = H;
          have = true;
        }
      }
      st->hi_star = best;
    }
    return;
  }

  if (stage == kL2) {
    if (st->n_neg > 0) select_step(st, 10, true, scratch);
    if (tid == 0) reset_neighbours(st);
    return;
  }

  if (stage == kLNb) {
    if (tid == 0) {
      // the list pass met only I_L's keys; the first pass kept the nearest
      // keys outside I_L, which lie below or above every key of I_L
      st->nb_below1 = max(st->nb_below1, st->l_nb_below1);
      if (st->l_nb_above_inv) st->nb_above = min(st->nb_above, ~st->l_nb_above_inv);
      // pieces at the ends of I_L: min{key > key(lo_min)}, 1 + max{key <= key(lo_max)}
      unsigned mp = st->l_mp_inv ? ~st->l_mp_inv : kNone;
      if (st->l_nb_above_inv) mp = min(mp, ~st->l_nb_above_inv);
      st->nb_mpiece = mp;
      st->nb_Mpiece1 = max(st->l_Mp1, st->l_nb_below1);
      const long long k = static_cast<long long>(st->k_bf16);
      const long long lb = static_cast<long long>(st->l_below), lin = static_cast<long long>(st->l_in);
      if (st->n_neg > 0 && k <= lb) {
        // C(lo_min) >= k already: |C - k| grows across I_L, so the bound is in
        // the piece that contains lo_min
        st->lo_star = lower_from_interval(a, st, -INFINITY, next_down(a.lo_min));
      } else if (st->n_neg > 0 && k > lb + lin) {
        // C(lo_max) < k: |C - k| shrinks across I_L, the piece containing lo_max
        st->lo_star = lower_from_interval(a, st, next_up(a.lo_max), INFINITY);
      } else if (st->n_neg > 0) {
        // minimisers of |C(L) - k|, C(L) = #{A<0 : r_fp8 <= L}, around u = r_(k),
        // which the select found inside I_L
        const float fu = __uint_as_float(st->u_key);
        const long long w_above = st->p_le - k, w_below = k - st->p_lt;
        const float z = st->nb_below1 ? __uint_as_float(st->nb_below1 - 1) : -INFINITY;
        const float w = st->nb_above != kNone ? __uint_as_float(st->nb_above) : INFINITY;
        float lo, hi;
        if (w_above < w_below) {
          lo = fu;
          hi = next_down(w);
        } else if (w_below < w_above) {
          lo = z;
          hi = next_down(fu);
        } else {
          lo = z;
          hi = next_down(w);
        }
        st->lo_star = lower_from_interval(a, st, lo, hi);
      }
      st->k_fp8 = 0;
      st->s_neg_fp = 0;
      st->below = 0;
      st->prefix = 0;
    }
    __syncthreads();
    zero_hist(st);
    return;
  }

  if (stage == kH0) {
    if (tid == 0) {
      sh_go = begin_upper(a, st);
      st->below = static_cast<long long>(st->h_below);  // P(hi_min): A>0 weight under I_H
    }
    __syncthreads();
    if (sh_go) select_step(st, 11, false, scratch);
    return;
  }

  if (stage == kH1 || stage == kH2) {
    if (tid == 0) sh_go = st->h_active && st->found;
    __syncthreads();
    if (sh_go) select_step(st, stage == kH1 ? 11 : 10, stage == kH2, scratch);
    if (stage == kH2 && tid == 0) {
      if (!st->found) st->u_key = kNone;
      reset_neighbours(st);
    }
    return;
  }

  if (stage == kHNb) {
    if (tid == 0 && st->h_active) {
      // minimisers of |P(H) D - X|, P(H) = sum_{A>0, r_fp8 < H} q, as a closed
      // float interval of H, from u and its positive-weight neighbours
      const U128 X{st->tgt_hi, st->tgt_lo};
      const unsigned long long D = static_cast<unsigned long long>(st->dmul);
      // the list pass met only I_H's keys; H0 kept the nearest q != 0 keys
      // outside I_H.  With u in I_H those below lie under u and those above
      // over it; with no u (P stays below the target) every key lies under it.
      if (st->found) {
        st->nb_below1 = max(st->nb_below1, st->h_nb_below1);
        if (st->h_nb_above_inv) st->nb_above = min(st->nb_above, ~st->h_nb_above_inv);
      } else {
        st->nb_below1 = max(st->nb_below1, max(st->h_nb_below1, st->h_top1));
      }
      // pieces at the ends of I_H: min{key >= key(hi_min), q > 0},
      // 1 + max{key < key(hi_max), q > 0}
      unsigned mp = st->h_mp_inv ? ~st->h_mp_inv : kNone;
      if (st->h_nb_above_inv) mp = min(mp, ~st->h_nb_above_inv);
      st->nb_mpiece = mp;
      st->nb_Mpiece1 = max(st->h_Mp1, st->h_nb_below1);
      const float z = st->nb_below1 ? __uint_as_float(st->nb_below1 - 1) : -INFINITY;
      const float w = st->nb_above != kNone ? __uint_as_float(st->nb_above) : INFINITY;
      float lo, hi;
      if (ge128(mul_u64(static_cast<unsigned long long>(st->h_below), D), X)) {
        // P(hi_min) D >= X already: the objective grows across I_H, so the
        // bound is in the piece that contains hi_min (P(H*) by the last pass)
        lo = -INFINITY;
        hi = next_down(a.hi_min);
      } else if (!st->found) {  // even all of P stays below the target
        lo = next_up(z);
        hi = INFINITY;
      } else {
        const float fu = __uint_as_float(st->u_key);
        const U128 above = sub128(mul_u64(static_cast<unsigned long long>(st->p_le), D), X);
        const U128 below = sub128(X, mul_u64(static_cast<unsigned long long>(st->p_lt), D));
        if (lt128(above, below)) {
          lo = next_up(fu);
          hi = w;
        } else if (lt128(below, above)) {
          lo = next_up(z);
          hi = fu;
        } else {
          lo = next_up(z);
          hi = w;
        }
      }
      st->hi_star = upper_from_interval(a, st, lo, hi);
      if (st->found) {
        // H* inside (z, u] or (u, w]: P(H*) is the select's p_lt or p_le
        const float H = st->hi_star, fu = __uint_as_float(st->u_key);
        if (H > fu && H <= w) {
          st->s_pos_fp = static_cast<unsigned long long>(st->p_le);
          st->p_known = 1;
        } else if (H <= fu && H > z) {
          st->s_pos_fp = static_cast<unsigned long long>(st->p_lt);
          st->p_known = 1;
        }
      }
    }
    return;
  }

  if (stage == kPFin) {
    if (tid == 0) write_result(a, st);
  }
}

__global__ void __launch_bounds__(1024) decide_kernel(Args a, int stage) {
  __shared__ long long sh_incl[kBuckets];
  decide_body(a, stage, sh_incl);
}

struct StageList {
  int n;
  int s[9];
};


// Grid-wide barrier of the one-launch kernel (all blocks co-resident: it is
// launched cooperatively).  Thread 0 of each block arrives on a counter; the
// last arrival opens the next generation.  The wait is bounded by the
// library's wait limit; false means it expired (the status word says so).
__device__ bool grid_barrier(State* st, uint64_t limit_ns, volatile int* sh_ok) {
  __syncthreads();
  if (gridDim.x == 1) return true;  // one block: the block barrier is the grid barrier
  if (threadIdx.x == 0) {
    bool ok = true;
    volatile unsigned* gen_p = &st->bar_gen;
    const unsigned gen = *gen_p;
    __threadfence();
    if (atomicAdd(&st->bar_count, 1u) == gridDim.x - 1) {
      st->bar_count = 0;
      __threadfence();
      atomicAdd(&st->bar_gen, 1u);
    } else {
      const uint64_t t0 = globaltimer_ns();
      while (*gen_p == gen) {
        if (globaltimer_ns() - t0 > limit_ns) {
          ok = false;
          flag(kErrTimeout);
          break;
        }
        __nanosleep(64);
      }
    }
    __threadfence();
    *sh_ok = ok;
  }
  __syncthreads();
  return *sh_ok != 0;
}

// Small and mid-size T: every pass and decision in one cooperative launch, so
// one launch replaces the 2 x 9 (or 2 x 3) launches of the grid path.  All
// blocks run each pass over their share of the tokens; block 0 then takes the
// decision while the others wait at the grid barrier.  The decide steps reuse
// the pass histogram's shared memory as scan scratch.
template <int G>
__global__ void __launch_bounds__(kCoopThreads) coop_kernel(Args a, StageList list, uint64_t limit_ns) {
  __shared__ ShHist sh;
  __shared__ float sh_cand[kBuckets];
  __shared__ int sh_ok;
  for (int i = 0; i < list.n; ++i) {
    pass_any<G>(a, list.s[i], sh, sh_cand);
    if (!grid_barrier(a.st, limit_ns, &sh_ok)) return;
    if (blockIdx.x == 0) decide_body(a, list.s[i], reinterpret_cast<long long*>(&sh));
    if (!grid_barrier(a.st, limit_ns, &sh_ok)) return;
  }
}

}  // namespace

// Launch shape of a call: one cooperative launch up to kCoopMaxT tokens, else
// pass / decide launches on up to four blocks of 256 per SM.  The interval
// lists get one segment per warp of the full passes, as long as the tokens
// that warp visits (its grid-stride steps of 32 lanes x G tokens, plus the
// T mod 4 tail that warp 0 takes).
struct CalibShape {
  bool coop;
  int blocks, threads;
  unsigned nseg, seg_cap;
};

CalibShape calib_shape(int64_t T, int G) {
  CalibShape c{};
  c.coop = T <= kCoopMaxT;
  if (c.coop) {
    int64_t nb = (T + kCoopTokensPerBlock - 1) / kCoopTokensPerBlock;
    nb = nb < 1 ? 1 : (nb > kCoopMaxBlocks ? kCoopMaxBlocks : nb);
    if (nb > sm_count()) nb = sm_count();
    c.blocks = static_cast<int>(nb);
    c.threads = kCoopThreads;
  } else {
    const int64_t want = (T + 4095) / 4096;
    const int64_t cap = static_cast<int64_t>(sm_count()) * 4;
    c.blocks = static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
    c.threads = 256;
  }
  c.nseg = static_cast<unsigned>(c.blocks) * static_cast<unsigned>(c.threads / 32);
  const int64_t ng = (T > 0 ? T : 0) / G;
  const int64_t per = static_cast<int64_t>(c.nseg) * 32;
  const int64_t steps = (ng + per - 1) / per;
  c.seg_cap = static_cast<unsigned>(steps * 32 * G + 32);
  return c;
}

size_t calib_state_bytes() { return align_up(sizeof(State), 256); }

// Workspace: the State, then (EXACT mode's interval lists) I_L keys, I_L
// segment fills, I_H keys, I_H q, I_H segment fills, for the larger of the
// two token groupings (4 tokens a lane with aligned inputs, else 1).
struct CalibLayout {
  size_t l_keys, l_cnt, h_keys, h_q, h_cnt, total;
  unsigned seg_cap;
};

CalibLayout calib_layout(int64_t T) {
  const CalibShape s1 = calib_shape(T, 1), s4 = calib_shape(T, 4);
  const unsigned cap = s1.seg_cap > s4.seg_cap ? s1.seg_cap : s4.seg_cap;
  const size_t n = static_cast<size_t>(s1.nseg) * cap;
  CalibLayout l{};
  size_t off = calib_state_bytes();
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, 256);
    return at;
  };
  l.l_keys = take(n * 4);
  l.l_cnt = take(static_cast<size_t>(s1.nseg) * 4);
  l.h_keys = take(n * 4);
  l.h_q = take(n * 8);
  l.h_cnt = take(static_cast<size_t>(s1.nseg) * 4);
  l.total = off;
  l.seg_cap = cap;
  return l;
}

size_t calib_workspace_bytes(int64_t T) { return calib_layout(T).total; }

cudaError_t launch_calibrate(const float* r_fp8, const float* r_bf16, const float* adv,
                             const uint8_t* mask, const float* coef, int64_t T, float eps_low,
                             float eps_high, const fp8rl_calib_opts& o, fp8rl_calib_result* result,
                             void* ws, cudaStream_t s) {
  Args a{};
  a.r_fp8 = r_fp8;
  a.r_bf16 = r_bf16;
  a.adv = adv;
  a.mask = mask;
  a.coef = coef;
  a.T = T;
  a.c_lo = 1.0f - eps_low;
  a.c_hi = 1.0f + eps_high;
  a.lo_min = static_cast<float>(o.lo_min);
  a.lo_max = static_cast<float>(o.lo_max);
  a.hi_min = static_cast<float>(o.hi_min);
  a.hi_max = static_cast<float>(o.hi_max);
  a.delta_lo = static_cast<float>(o.delta_lo);
  a.delta_hi = static_cast<float>(o.delta_hi);
  a.lo_old = o.lo_old;
  a.hi_old = o.hi_old;
  a.grid_mode = o.mode == FP8RL_CALIB_GRID;
  a.lo_grid0 = o.lo_min;
  a.hi_grid0 = o.hi_min;
  a.step = o.step;
  a.n_lcand = a.grid_mode ? static_cast<int>(std::llround((o.lo_max - o.lo_min) / o.step)) + 1 : 0;
  a.n_hcand = a.grid_mode ? static_cast<int>(std::llround((o.hi_max - o.hi_min) / o.step)) + 1 : 0;
  a.st = static_cast<State*>(ws);
  a.out = result;
  const CalibLayout lay = calib_layout(T);
  char* base = static_cast<char*>(ws);
  a.l_keys = reinterpret_cast<unsigned*>(base + lay.l_keys);
  a.l_cnt = reinterpret_cast<unsigned*>(base + lay.l_cnt);
  a.h_keys = reinterpret_cast<unsigned*>(base + lay.h_keys);
  a.h_q = reinterpret_cast<long long*>(base + lay.h_q);
  a.h_cnt = reinterpret_cast<unsigned*>(base + lay.h_cnt);
  a.seg_cap = lay.seg_cap;

  cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(State), s);
  if (e != cudaSuccess) return e;
  auto al = [](const void* p, uintptr_t n) { return (reinterpret_cast<uintptr_t>(p) & (n - 1)) == 0; };
  const bool vec = al(r_fp8, 16) && al(r_bf16, 16) && al(adv, 16) && al(coef, 16) && al(mask, 4);
  const CalibShape sh = calib_shape(T, vec ? 4 : 1);
  a.nseg = sh.nseg;  // the layout's segment capacity covers either grouping
  const int stages_exact[] = {kPrep, kSums, kL2, kLNb, kH0, kH1, kH2, kHNb, kPFin};
  const int stages_grid[] = {kPrep, kSums, kPFin};
  const int* stages = a.grid_mode ? stages_grid : stages_exact;
  const int n = a.grid_mode ? 3 : 9;
  if (sh.coop) {
    StageList list{};
    list.n = n;
    for (int i = 0; i < n; ++i) list.s[i] = stages[i];
    uint64_t limit = wait_limit_ns();
    void* args[] = {&a, &list, &limit};
    const void* fn = vec ? reinterpret_cast<const void*>(&coop_kernel<4>)
                         : reinterpret_cast<const void*>(&coop_kernel<1>);
    return cudaLaunchCooperativeKernel(fn, dim3(static_cast<unsigned>(sh.blocks)), dim3(sh.threads), args, 0, s);
  }
  for (int i = 0; i < n; ++i) {
    if (vec) launch_pass<4>(a, stages[i], sh.blocks, s);
    else launch_pass<1>(a, stages[i], sh.blocks, s);
    decide_kernel<<<1, 1024, 0, s>>>(a, stages[i]);
  }
  return cudaGetLastError();
}

uint32_t calib_status_take() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, d_status, sizeof(v)) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(d_status, &z, sizeof(z));
  return v;
}

}  // namespace fp8rl
