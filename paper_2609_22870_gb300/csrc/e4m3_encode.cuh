// E4M3 encoding of bf16 data, Q_FP8(fl32(x / S)) (Section 2.2 quantiser:
// divide by the block scale, round to nearest even, saturate to +-448), in
// packed pair arithmetic.
//
// The quotient fl32(x / S) is computed without a division by Markstein's
// correction (P. Markstein, "Computation of elementary functions on the IBM
// RISC System/6000 processor", IBM J. Res. Dev. 34(1), 1990; also J.-M. Muller
// et al., Handbook of Floating-Point Arithmetic, division by FMA): with
// y = RN(1 / S) and q = RN(x * y) within one ulp of x / S, the remainder
// r = x - q * S is exact in one FMA and RN(q + r * y) is the correctly rounded
// quotient, provided nothing underflows.  Here it runs on negated values, so
// that the sign of x = -0 survives and no negation is needed per element:
//   qn = RN(x * (-y)),  r = RN(x + qn * S) = x - q * S,  d = RN(qn - r * y) = -RN(x / S),
// and the E4M3 code of -d is the code of d with its sign bit flipped (E4M3 is
// sign-magnitude and round-to-nearest-even with saturation is symmetric).
//
// Underflow is excluded by scale: with S >= 2^-80 every quotient that can
// round to a non-zero code (|x / S| >= 2^-10) has a remainder on a grid no
// finer than 2^-149, so r stays exact; smaller S (amax below 448 * 2^-80) take
// the correctly rounded division instead.  The largest S a finite bf16 amax
// gives (3.39e38 / 448 < 2^120) keeps y = RN(1 / S) a normal number.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp8.h>
#include <stdint.h>

namespace fp8rl {

constexpr float kE4M3Max = 448.f;
constexpr float kMarksteinMinScale = 8.271806125530277e-25f;  // 2^-80

// A pair of floats in one 64-bit register pair, lane 0 in the low half.
__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}

// Two bf16 in one 32-bit word (element 0 in the low half) as two floats.
__device__ __forceinline__ uint64_t bf16x2_to_f32x2(uint32_t v) {
  return f32x2(__uint_as_float(v << 16), __uint_as_float(v & 0xFFFF0000u));
}

// m = max(|m|, |v|) per bf16 lane, NaN-propagating.  The sign of the result
// is the XOR of the operand signs: callers take |m| at the end.
__device__ __forceinline__ uint32_t amax_bf16x2(uint32_t m, uint32_t v) {
  uint32_t d;
  asm("max.NaN.xorsign.abs.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(m), "r"(v));
  return d;
}

// Largest |x| of a packed bf16x2 running maximum, as a float; +inf or NaN
// when any reduced value was not finite.
__device__ __forceinline__ float amax_of(uint32_t m) {
  const uint32_t a = m & 0x7FFF7FFFu;
  const uint32_t hi = a >> 16, lo = a & 0xFFFFu;
  return __uint_as_float((hi > lo ? hi : lo) << 16);
}

// The smallest power of two not below t (t > 0; finite t < 2^119 here).
// +inf and NaN (a block with a non-finite input) come back unchanged, so the
// stored scale shows the bad block as in the paper-scale mode.
__device__ __forceinline__ float pow2_ceil(float t) {
  const uint32_t b = __float_as_uint(t);
  const uint32_t ex = b >> 23, man = b & 0x7FFFFFu;
  if (ex == 0xFFu || man == 0) return t;               // inf / NaN, or a power of two
  if (ex != 0) return __uint_as_float((ex + 1) << 23);  // next binade
  const int h = 31 - __clz(man);                       // subnormal: highest set bit
  return man == (1u << h) ? t : __uint_as_float(1u << (h + 1));
}

// A power-of-two scale that the FP8 backward forms itself, raised to 2^-127
// (E8M0's smallest scale, a float32 subnormal) where it falls below; s >= 0
// or NaN, which stays NaN.
__device__ __forceinline__ float e8m0_floor(float s) {
  return __float_as_uint(s) < 0x00400000u ? __uint_as_float(0x00400000u) : s;
}

// S = fl32(amax / 448), 1 when amax == 0 (an all-zero block keeps S = 1);
// with pow2 (UE8M0 scales) rounded up to a power of two, so that |x / S|
// stays within 448 and x / S is exact.
__device__ __forceinline__ float e4m3_scale(float amax, bool pow2) {
  const float s = amax == 0.f ? 1.f : __fdiv_rn(amax, kE4M3Max);
  return pow2 ? pow2_ceil(s) : s;
}

// Per-scale constants of the packed encoder.
struct E4M3Enc {
  uint64_t s2;    // {S, S}
  uint64_t ny2;   // {-RN(1/S), -RN(1/S)}
  float s;
  bool divide;    // S below the Markstein range: use the division
};

__device__ __forceinline__ E4M3Enc e4m3_encoder(float s) {
  E4M3Enc e;
  e.s = s;
  e.divide = !(s >= kMarksteinMinScale);
  const float ny = -__frcp_rn(s);
  e.s2 = f32x2(s, s);
  e.ny2 = f32x2(ny, ny);
  return e;
}

// -RN(x / S) for both lanes of a pair.
__device__ __forceinline__ uint64_t neg_quotient2(uint64_t x2, const E4M3Enc& e) {
  uint64_t qn, r, d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(qn) : "l"(x2), "l"(e.ny2));
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(qn), "l"(e.s2), "l"(x2));
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(r), "l"(e.ny2), "l"(qn));
  return d;
}

// E4M3 codes (satfinite, round to nearest even) of both lanes, lane 0 in the
// low byte.
__device__ __forceinline__ uint32_t cvt_e4m3x2(uint64_t v2) {
  float lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v2));
  return static_cast<uint32_t>(
      __nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE, __NV_E4M3));
}

// Codes Q_FP8(fl32(x_i / S)) of 8 bf16 (a 16-byte group), byte i = element i.
__device__ __forceinline__ uint2 e4m3_encode8(const uint4& v, const E4M3Enc& e) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t c[4];
  if (!e.divide) {
#pragma unroll
    for (int i = 0; i < 4; ++i) c[i] = cvt_e4m3x2(neg_quotient2(bf16x2_to_f32x2(w[i]), e));
    return make_uint2((c[0] | (c[1] << 16)) ^ 0x80808080u, (c[2] | (c[3] << 16)) ^ 0x80808080u);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float lo = __fdiv_rn(__uint_as_float(w[i] << 16), e.s);
    const float hi = __fdiv_rn(__uint_as_float(w[i] & 0xFFFF0000u), e.s);
    c[i] = static_cast<uint32_t>(
        __nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE, __NV_E4M3));
  }
  return make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
}

// Running |x| maximum of a 16-byte group of 8 bf16.
__device__ __forceinline__ uint32_t amax_bf16x8(uint32_t m, const uint4& v) {
  return amax_bf16x2(amax_bf16x2(amax_bf16x2(amax_bf16x2(m, v.x), v.y), v.z), v.w);
}

}  // namespace fp8rl
