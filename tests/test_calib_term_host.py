"""Host check of the calibration kernel's Eq. 5 term arithmetic (no GPU).

The kernel forms q = RNE(fl64(fl64(c r) A) 2^s) in two ways: a float32 path
(error-free products, a power-of-two scale, rounding to the nearest integer
when the value is more than 2^-9 from a tie) and the exact integer path for
everything else.  Both are plain arithmetic, so this test compiles the two
device functions from csrc/calib.cu as host C++ (with host stand-ins for the
bit-cast and 64-bit multiply intrinsics) and compares them, and the integer
path with the host's IEEE float64 arithmetic (llrint(ldexp(fl64(fl64(c r) A),
s)), round half to even), on seeded random triples: realistic coefficients,
wide exponent ranges, values planted on and next to rounding ties, raw bit
patterns, and large values (2^30 .. 2^35) within 2^-12 of a tie, where the
53-bit rounding and the float32 path's error come nearest its 2^-9 margin.
"""

import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CALIB = os.path.join(ROOT, "paper_2609_22870_gb300", "csrc", "calib.cu")

SHIMS = r"""
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <cmath>
#include <cstdio>
#include <random>
static inline unsigned __float_as_uint(float f) { unsigned u; memcpy(&u, &f, 4); return u; }
static inline float __int_as_float(int i) { float f; memcpy(&f, &i, 4); return f; }
static inline unsigned long long __umul64hi(unsigned long long a, unsigned long long b) {
  return (unsigned long long)(((unsigned __int128)a * b) >> 64);
}
static inline int __clzll(long long x) { return x == 0 ? 64 : __builtin_clzll((unsigned long long)x); }
"""

MAIN = r"""
static bool ref_q(float c, float r, float a, int s, long long& q) {
  const double e = ((double)c * (double)r) * (double)a;  // c r exact; one rounding
  const double x = std::ldexp(e, s);
  if (!(std::fabs(x) < 9.2e18)) return false;
  q = std::llrint(x);
  return true;
}
int main(int argc, char** argv) {
  const long long N = atoll(argv[1]);
  std::mt19937_64 g(20261202);
  std::normal_distribution<double> nd(0.0, 1.0);
  std::uniform_real_distribution<double> ud(0.0, 1.0);
  long long n = 0, fast = 0, bad_fast = 0, bad_exact = 0, ties = 0;
  for (long long it = 0; it < N; ++it) {
    const int mode = (int)(it % 4);
    float c, r, a;
    int s;
    if (mode == 0) {  // pi_sampler-like coefficients at the shifts of 2^20..2^27 tokens
      c = (float)std::exp(-11.0 + 2.0 * nd(g)); r = (float)std::exp(0.1 * nd(g)); a = (float)nd(g);
      s = 26 + (int)(g() % 16);
    } else if (mode == 1) {  // wide exponent ranges
      c = (float)std::ldexp(1.0 + ud(g), (int)(g() % 200) - 150);
      r = (float)std::ldexp(1.0 + ud(g), (int)(g() % 60) - 30);
      a = (float)(nd(g) * std::ldexp(1.0, (int)(g() % 40) - 20));
      s = (int)(g() % 300) - 150;
    } else if (mode == 2) {  // on and next to the ties k + 1/2
      r = (float)(1.0 + ud(g)); a = (float)((g() & 1 ? -1 : 1) * (1.0 + ud(g))); s = (int)(g() % 34);
      const double d = (g() & 1 ? 1 : -1) * std::ldexp(1.0, -(int)(g() % 24));
      const double V = std::floor(ud(g) * 1000.0) + 0.5 + ((g() & 3) ? d : 0.0);
      c = (float)std::fabs(V / ((double)r * a * std::ldexp(1.0, s)));
      if (g() % 8 == 0) { r = 1.0f; a = a < 0 ? -1.0f : 1.0f; c = (float)std::ldexp(std::floor(V) + 0.5, -s); }
    } else {  // raw bit patterns (c, r >= 0)
      unsigned u1 = (unsigned)g() & 0x7FFFFFFFu, u2 = (unsigned)g() & 0x7FFFFFFFu, u3 = (unsigned)g();
      memcpy(&c, &u1, 4); memcpy(&r, &u2, 4); memcpy(&a, &u3, 4);
      s = (int)(g() % 400) - 200;
      if (!std::isfinite(c) || !std::isfinite(r) || !std::isfinite(a)) continue;
    }
    ++n;
    const long long qe = fixed_term_exact(c, r, a, s);
    long long qr;
    if (ref_q(c, r, a, s, qr) && qr != qe) ++bad_exact;
    if (mode == 2) {
      const double x = std::ldexp(std::fabs(((double)c * r) * a), s);
      if (std::fabs(x - std::floor(x) - 0.5) < std::ldexp(1.0, -8)) ++ties;
    }
    long long qf;
    if (fixed_term_fast(c, r, a, s, qf)) { ++fast; if (qf != qe) ++bad_fast; }
  }
  // large values within 2^-12 of a half-integer, where the 53-bit rounding of
  // the product and the float32 estimate's error both come near the margin
  long long big = 0, draws = 0, near_taken = 0;
  while (big < 3000 && draws < 200000000LL) {
    ++draws;
    const float c = (float)std::ldexp(1.0 + ud(g), -16 - (int)(g() % 4));
    const float r = (float)(0.5 + ud(g));
    const float a = (float)((g() & 1 ? -1 : 1) * (0.5 + ud(g)));
    const int s = 46 + (int)(g() % 5);
    const double x = std::ldexp(std::fabs(((double)c * r) * a), s);
    if (!(x >= 0x1p30 && x < 0x1p35) || std::fabs(x - std::floor(x) - 0.5) >= std::ldexp(1.0, -12)) continue;
    ++big; ++n;
    const long long qe = fixed_term_exact(c, r, a, s);
    long long qr;
    if (ref_q(c, r, a, s, qr) && qr != qe) ++bad_exact;
    long long qf;
    if (fixed_term_fast(c, r, a, s, qf)) { ++fast; ++near_taken; if (qf != qe) ++bad_fast; }
  }
  printf("%lld %lld %lld %lld %lld %lld %lld\n", n, fast, bad_fast, bad_exact, ties, big, near_taken);
  return 0;
}
"""


def test_term_fast_path_agrees_with_integer_path_and_float64(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    src = open(CALIB).read()
    i = src.index("// |x| = m 2^e with an integer significand m < 2^24.")
    j = src.index("__device__ __forceinline__ bool digit_match")
    body = src[i:j].replace("__device__ __forceinline__", "static inline")
    k = re.search(r"constexpr int kEBias = \d+;", src)
    cpp = tmp_path / "term.cpp"
    cpp.write_text(SHIMS + k.group(0) + "\n" + body + MAIN)
    exe = tmp_path / "term"
    subprocess.run([cxx, "-O2", "-std=c++17", "-o", str(exe), str(cpp)], check=True, capture_output=True)
    out = subprocess.run([str(exe), "4000000"], check=True, capture_output=True, text=True).stdout.split()
    n, fast, bad_fast, bad_exact, ties, big, near_taken = (int(x) for x in out)
    assert bad_fast == 0 and bad_exact == 0
    # values within 2^-12 of a tie never take the float32 path: its margin
    # (2^-9) exceeds its error bound (2^-10), which is what makes it exact
    assert near_taken == 0
    # both paths, the small ties and the large near-ties were exercised
    assert fast > n // 4 and ties > n // 16 and big == 3000
