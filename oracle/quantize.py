"""Scaled FP8 quantisation (Eq. 3, §2.2) -- oracle side.

Test infrastructure only (see ``oracle/__init__.py``).

Eq. 3: S_X = max|X| / F_max,  X_hat = Q_FP8(X / S_X),  X_tilde = S_X * X_hat,
with F_max = 448 for E4M3.  §2.2 names three granularities for max|X|:
tensorwise (one S for the whole tensor), rowwise (one S per row) and
blockwise (one S per sub-block, e.g. 128x128).

Readings taken where the paper is silent:

* S is the float32 quotient fl32(amax / 448); amax is the exact maximum of |x|
  over the block (bf16 inputs are exact in float32).  amax == 0 gives S = 1 and
  all-zero codes.
* The quotient x / S is the correctly rounded float32 value fl32(x / S) (not
  x * (1/S)); Q_FP8 is then applied to that float32 (two roundings, as a
  float32 -> E4M3 conversion does).
* "rowwise" for the lm_head GEMM operands means one scale per token row of the
  hidden states h[T][H] and one per vocabulary row (output channel) of
  W[V][H].
* "blockwise" is 1x128 for the activations h (one scale per token per 128
  hidden columns) and 128x128 for the weight W.  A tail block of W along V
  (V not a multiple of 128) takes its amax over the rows that exist; the
  hidden size must be a multiple of 128 in block mode.

Power-of-two (UE8M0) variant, outside the paper (its S is amax / 448): the
scale format that the hardware's block-scaled MMA takes.  S is rounded up to
the smallest power of two not below fl32(amax / 448), so |x / S| <= 448 still
holds and x / S is exact; amax == 0 gives S = 1.  Where the scales are formed
by the FP8 backward itself (not given as input), a floor keeps them inside
E8M0's range: S = max(that power of two, 2^-127), so a block of tiny values
(e.g. a row of dLoss/dlogits whose probabilities underflow) still has a scale
the MMA takes; x / S stays exact.

Scales are returned in their natural shapes:
  tensor: (1,);  row: (rows,);  act block: (rows, cols/128);
  weight block: (ceil(rows/128), cols/128).
"""

import numpy as np

from . import e4m3

TENSOR, ROWWISE, BLOCK = 0, 1, 2
ACT, WEIGHT = 0, 1
E8M0_MIN = 2.0 ** -127  # the smallest E8M0 scale (biased exponent 0)
BLOCK_K = 128  # block edge along the hidden (reduction) dimension
BLOCK_W = 128  # block edge of the weight along the vocabulary dimension


def scale_from_amax(amax):
    """S = fl32(amax / F_max) (Eq. 3); 1.0 where amax == 0."""
    amax = np.asarray(amax, dtype=np.float32)
    s = (amax / np.float32(e4m3.E4M3_MAX)).astype(np.float32)
    return np.where(amax == 0, np.float32(1.0), s).astype(np.float32)


def pow2_scale_from_amax(amax):
    """S = 2^ceil(log2(fl32(amax / F_max))); 1.0 where amax == 0."""
    s = scale_from_amax(amax).astype(np.float64)
    m, e = np.frexp(s)  # s = m 2^e, m in [0.5, 1)
    p = np.where(m == 0.5, s, np.ldexp(1.0, e))
    return p.astype(np.float32)


def _encode_block(x, s):
    """Q_FP8(fl32(x / S)) for a block x with its scale s (broadcastable)."""
    q = (x.astype(np.float32) / np.asarray(s, dtype=np.float32)).astype(np.float32)
    return e4m3.encode(q)


def quantize(x, gran, role=ACT, pow2=False, scale_floor=0.0):
    """Quantise a 2-D float32 array (bf16-valued) at the given granularity.

    Returns (codes uint8 [rows][cols], scales float32 in natural shape).
    ``pow2`` selects the power-of-two (UE8M0) scales; ``scale_floor`` raises
    every scale below it to it (E8M0_MIN for the backward's own scales).
    """
    base = pow2_scale_from_amax if pow2 else scale_from_amax

    def scale_from(amax):
        return np.maximum(base(amax), np.float32(scale_floor)).astype(np.float32)

    x = np.asarray(x, dtype=np.float32)
    if x.ndim != 2:
        raise ValueError("quantize: 2-D input expected")
    rows, cols = x.shape
    if not np.all(np.isfinite(x)):
        raise ValueError("quantize: non-finite input")
    if gran == TENSOR:
        s = scale_from(np.max(np.abs(x)) if x.size else np.float32(0))
        s = np.asarray(s, dtype=np.float32).reshape(1)
        return _encode_block(x, s[0]), s
    if gran == ROWWISE:
        amax = np.max(np.abs(x), axis=1) if cols else np.zeros(rows, np.float32)
        s = scale_from(amax)
        return _encode_block(x, s[:, None]), s
    if gran != BLOCK:
        raise ValueError("quantize: unknown granularity")
    if cols % BLOCK_K:
        raise ValueError("quantize: block mode needs cols % 128 == 0")
    nkb = cols // BLOCK_K
    if role == ACT:
        xb = x.reshape(rows, nkb, BLOCK_K)
        s = scale_from(np.max(np.abs(xb), axis=2))  # (rows, nkb)
        codes = _encode_block(xb, s[:, :, None]).reshape(rows, cols)
        return codes, s
    # weight: 128 x 128 blocks, tail rows along V allowed; one 128-row strip
    # (all its blocks) at a time
    nrb = (rows + BLOCK_W - 1) // BLOCK_W
    s = np.empty((nrb, nkb), dtype=np.float32)
    codes = np.empty((rows, cols), dtype=np.uint8)
    for rb in range(nrb):
        r0, r1 = rb * BLOCK_W, min(rows, (rb + 1) * BLOCK_W)
        strip = x[r0:r1].reshape(r1 - r0, nkb, BLOCK_K)
        sb = scale_from(np.max(np.abs(strip), axis=(0, 2)))  # (nkb,)
        s[rb] = sb
        codes[r0:r1] = _encode_block(strip, sb[None, :, None]).reshape(r1 - r0, cols)
    return codes, s


def dequantize(codes, scales, gran, role=ACT):
    """X_tilde = S * X_hat (Eq. 3) in float64, scales in natural shape."""
    v = e4m3.decode(codes)
    rows, cols = v.shape
    s = np.asarray(scales, dtype=np.float64)
    if gran == TENSOR:
        return v * s.reshape(-1)[0]
    if gran == ROWWISE:
        return v * s[:, None]
    nkb = cols // BLOCK_K
    if role == ACT:
        return (v.reshape(rows, nkb, BLOCK_K) * s[:, :, None]).reshape(rows, cols)
    srow = np.repeat(s, BLOCK_W, axis=0)[:rows]  # (rows, nkb)
    return (v.reshape(rows, nkb, BLOCK_K) * srow[:, :, None]).reshape(rows, cols)
