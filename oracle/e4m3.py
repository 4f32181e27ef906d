"""OCP FP8 E4M3 ("fn" variant) decode / encode -- oracle side.

Test infrastructure only (see ``oracle/__init__.py``).

The paper's Q_FP8 (Eq. 3, §2.2) is "rounding and clamping to the FP8
representable set".  The FP8 format used on the hot path is E4M3 as defined by
the OCP 8-bit floating point specification:

* bit 7 sign, bits 6..3 exponent (bias 7), bits 2..0 mantissa;
* exponent field 0: subnormal, value = m * 2**-9;
* otherwise value = (1 + m/8) * 2**(e - 7);
* S.1111.111 (0x7F / 0xFF) is NaN; there is no infinity; the largest finite
  magnitude is 0b1111.110 = 448.

Reading taken for Q_FP8: round to nearest, ties to even mantissa, applied to
the float32 value x/S; magnitudes at or above 448 saturate to +-448 (there is
no infinity to overflow into); the sign is kept, so -0.0 encodes as 0x80.
"""

import numpy as np

E4M3_MAX = 448.0
NAN_CODES = (0x7F, 0xFF)


def decode(codes):
    """Value of each E4M3 code as float64 (NaN for 0x7F / 0xFF)."""
    c = np.asarray(codes, dtype=np.uint8).astype(np.int64)
    sign = np.where(c & 0x80, -1.0, 1.0)
    e = (c >> 3) & 0xF
    m = c & 0x7
    sub = m.astype(np.float64) * 2.0 ** -9
    norm = (1.0 + m.astype(np.float64) / 8.0) * np.exp2(e.astype(np.float64) - 7.0)
    val = sign * np.where(e == 0, sub, norm)
    val = np.where((e == 15) & (m == 7), np.nan, val)
    return val


# The 127 non-negative finite codes 0x00..0x7E decode to strictly increasing
# magnitudes, so a code's position in this table is the code itself.
_POS_CODES = np.arange(0x7F, dtype=np.uint8)
_POS_VALUES = decode(_POS_CODES)
assert np.all(np.diff(_POS_VALUES) > 0)


def encode(q):
    """Encode float32 values to E4M3 codes: RNE, ties to even, satfinite.

    ``q`` must be finite.  The nearest representable magnitude is found by an
    exact float64 comparison of the two neighbouring table entries; float64
    holds every float32 and every E4M3 value, and their differences, exactly.
    """
    q = np.asarray(q, dtype=np.float32)
    if not np.all(np.isfinite(q)):
        raise ValueError("E4M3 encode: non-finite input")
    a = np.abs(q).astype(np.float64)
    neg = np.signbit(q)
    idx = np.searchsorted(_POS_VALUES, a, side="right") - 1  # lo <= a
    idx = np.clip(idx, 0, 0x7E)
    lo = _POS_VALUES[idx]
    hi = _POS_VALUES[np.minimum(idx + 1, 0x7E)]
    d_lo = a - lo
    d_hi = hi - a
    up = (d_hi < d_lo) | ((d_hi == d_lo) & (idx % 2 == 1))
    code = np.where(up, idx + 1, idx)
    code = np.where(a >= E4M3_MAX, 0x7E, code)  # saturate (no infinity)
    code = code.astype(np.uint8) | np.where(neg, 0x80, 0).astype(np.uint8)
    return code.astype(np.uint8)
