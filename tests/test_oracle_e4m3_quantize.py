"""Pins for the oracle's E4M3 codec and scaled quantisation (Eq. 3, §2.2).

The oracle is checked against things other than itself: the OCP E4M3 code
table, PyTorch's float32 -> float8_e4m3fn cast (a library routine that rounds
to nearest even in range), closed forms for the scale and for the amax element,
and the E4M3 rounding error bound.
"""

import os

import numpy as np
import pytest
import torch

from oracle import e4m3
from oracle import quantize as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _ocp_table():
    rows = []
    for line in open(os.path.join(GOLDEN, "e4m3_ocp.txt")):
        line = line.split("#")[0].strip()
        if line:
            code, val = line.split()
            rows.append((int(code, 16), float(val)))
    return rows


def test_decode_matches_ocp_table():
    for code, val in _ocp_table():
        got = e4m3.decode(np.array([code], np.uint8))[0]
        if np.isnan(val):
            assert np.isnan(got), hex(code)
        else:
            assert got == val and np.signbit(got) == np.signbit(val), hex(code)


def test_round_trip_all_finite_codes():
    codes = np.array([c for c in range(256) if c not in e4m3.NAN_CODES], np.uint8)
    assert codes.size == 254
    vals = e4m3.decode(codes).astype(np.float32)
    assert np.array_equal(e4m3.encode(vals), codes)


def test_encode_matches_torch_cast_in_range():
    rng = np.random.default_rng(7)
    # random magnitudes across the whole exponent range, plus exact midpoints
    x = (rng.standard_normal(400_000) * np.exp2(rng.integers(-14, 9, 400_000))).astype(np.float32)
    x = np.clip(x, -448, 448)
    finite = e4m3.decode(np.arange(0x7F, dtype=np.uint8))
    mids = ((finite[1:] + finite[:-1]) / 2).astype(np.float32)
    x = np.concatenate([x, mids, -mids, np.nextafter(mids, 0), np.nextafter(mids, 1000)])
    ref = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(e4m3.encode(x), ref)


def test_ties_to_even_and_saturation():
    # 1.0625 lies halfway between 1.0 (0x38) and 1.125 (0x39): even -> 0x38.
    # 1.1875 lies halfway between 1.125 (0x39) and 1.25 (0x3A): even -> 0x3A.
    # 2^-10 lies halfway between 0 and the min subnormal: even -> 0x00.
    x = np.array([1.0625, 1.1875, 2.0 ** -10, 464.0, 448.5, 1e6, -1e6, -0.0], np.float32)
    assert e4m3.encode(x).tolist() == [0x38, 0x3A, 0x00, 0x7E, 0x7E, 0x7E, 0xFE, 0x80]
    with pytest.raises(ValueError):
        e4m3.encode(np.array([np.nan], np.float32))


def test_scale_closed_form():
    assert Q.scale_from_amax(np.float32(448.0)) == np.float32(1.0)
    assert Q.scale_from_amax(np.float32(0.0)) == np.float32(1.0)
    assert Q.scale_from_amax(np.float32(3.5)) == np.float32(3.5) / np.float32(448.0)
    codes, s = Q.quantize(np.zeros((3, 256), np.float32), Q.BLOCK, Q.ACT)
    assert np.all(codes == 0) and np.all(s == 1.0)


def _bf16(a):
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).float().numpy()


@pytest.mark.parametrize("gran,role", [(Q.TENSOR, Q.ACT), (Q.ROWWISE, Q.ACT), (Q.ROWWISE, Q.WEIGHT),
                                       (Q.BLOCK, Q.ACT), (Q.BLOCK, Q.WEIGHT)])
def test_amax_element_maps_to_fmax_and_error_bound(gran, role):
    rng = np.random.default_rng(11 + gran)
    x = _bf16(rng.standard_normal((300, 384)) * rng.choice([0.02, 1.0, 30.0], size=(300, 1)))
    codes, s = Q.quantize(x, gran, role)
    xt = Q.dequantize(codes, s, gran, role)
    # every block's largest |x| encodes to +-448
    if gran == Q.TENSOR:
        blocks = [(slice(None), slice(None))]
    elif gran == Q.ROWWISE:
        blocks = [(slice(r, r + 1), slice(None)) for r in range(300)]
    elif role == Q.ACT:
        blocks = [(slice(r, r + 1), slice(k, k + 128)) for r in range(0, 300, 37) for k in (0, 128, 256)]
    else:
        blocks = [(slice(r, min(300, r + 128)), slice(k, k + 128)) for r in (0, 128, 256) for k in (0, 128, 256)]
    for b in blocks:
        xb, cb = x[b], codes[b]
        i = np.unravel_index(np.argmax(np.abs(xb)), xb.shape)
        if xb[i] != 0:
            assert cb[i] in (0x7E, 0xFE)
            assert (cb[i] == 0xFE) == (xb[i] < 0)
    # RNE error bound of E4M3 relative to the scaled value: half a quantum
    s_full = Q.dequantize(np.full(codes.shape, 0x38, np.uint8), s, gran, role)  # S broadcast
    q = x / s_full
    e = np.floor(np.log2(np.maximum(np.abs(q), 2.0 ** -6)))
    half_quantum = np.exp2(e - 3) / 2  # 3 mantissa bits; subnormal quantum 2^-9
    assert np.all(np.abs(xt / s_full - q) <= half_quantum * (1 + 1e-6) + 1e-12)


def test_tensor_equals_single_block_and_row_equals_per_row_tensor():
    rng = np.random.default_rng(3)
    x = _bf16(rng.standard_normal((1, 128)))
    ct, st = Q.quantize(x, Q.TENSOR)
    cb, sb = Q.quantize(x, Q.BLOCK, Q.ACT)
    assert np.array_equal(ct, cb) and st[0] == sb[0, 0]
    x = _bf16(rng.standard_normal((5, 256)) * 3)
    cr, sr = Q.quantize(x, Q.ROWWISE, Q.ACT)
    for r in range(5):
        c1, s1 = Q.quantize(x[r:r + 1], Q.TENSOR)
        assert np.array_equal(c1[0], cr[r]) and s1[0] == sr[r]


def test_weight_block_tail_rows():
    rng = np.random.default_rng(5)
    x = _bf16(rng.standard_normal((130, 128)))
    c, s = Q.quantize(x, Q.BLOCK, Q.WEIGHT)
    assert s.shape == (2, 1)
    c2, s2 = Q.quantize(x[128:], Q.TENSOR)
    assert np.array_equal(c[128:], c2) and s[1, 0] == s2[0]


# ---- power-of-two (UE8M0) scales ----------------------------------------------

def test_pow2_scale_closed_form():
    amax = np.array([0.0, 448.0, 224.0, 448.0 * 3, 1.0, 2.0 ** -130, 300.0], np.float32)
    s = Q.pow2_scale_from_amax(amax)
    plain = Q.scale_from_amax(amax).astype(np.float64)
    assert s[0] == 1.0 and s[1] == 1.0 and s[2] == 0.5 and s[3] == 4.0
    m, _ = np.frexp(s[1:].astype(np.float64))
    assert np.all(m == 0.5)  # powers of two
    assert np.all(s[1:] >= plain[1:]) and np.all(s[1:] < 2 * plain[1:])


def _per_element(s, gran, role, rows, cols):
    """Scales broadcast to the element grid."""
    s = np.asarray(s, np.float64)
    if gran == Q.TENSOR:
        return np.full((rows, cols), s[0])
    if gran == Q.ROWWISE:
        return np.repeat(s[:, None], cols, axis=1)
    if role == Q.ACT:
        return np.repeat(s, 128, axis=1)
    return np.repeat(np.repeat(s, 128, axis=0)[:rows], 128, axis=1)


@pytest.mark.parametrize("gran,role", [(Q.TENSOR, Q.ACT), (Q.ROWWISE, Q.ACT), (Q.BLOCK, Q.ACT),
                                       (Q.BLOCK, Q.WEIGHT)])
def test_pow2_quantize_bounds_and_agreement(gran, role):
    rng = np.random.default_rng(50 + gran + role)
    rows, cols = 300, 256
    x = (rng.standard_normal((rows, cols)) * np.exp2(rng.integers(-8, 8, (rows, 1)))).astype(np.float32)
    codes, s = Q.quantize(x, gran, role, pow2=True)
    m, _ = np.frexp(s.astype(np.float64))
    assert np.all(m == 0.5)
    S = _per_element(s, gran, role, rows, cols)
    # x / S is exact and at most 448 in magnitude, so each code is x / S rounded
    # to nearest: within half an E4M3 quantum (2^-4 relative in the normal
    # range, 2^-10 absolute below 2^-6)
    assert np.all(np.abs(x / S) <= 448)
    err = np.abs(Q.dequantize(codes, s, gran, role) - x.astype(np.float64))
    assert np.all(err <= np.maximum(np.abs(x) * 2.0 ** -4, S * 2.0 ** -10))
    # where the paper's S is already a power of two the codes agree bit for bit:
    # give every row / block an element of magnitude 448 * 2^k
    # (rows scaled into [-1, 1]; every maximum over a row, block or the tensor is
    # then one of the planted values)
    y = (x / np.max(np.abs(x), axis=1, keepdims=True)).astype(np.float32)
    for c0 in range(0, cols, 128):
        y[:, c0] = np.float32(448.0) * np.exp2(rng.integers(-2, 6, rows)).astype(np.float32)
    pc, ps = Q.quantize(y, gran, role, pow2=True)
    qc, qs = Q.quantize(y, gran, role)
    assert np.array_equal(ps, qs) and np.array_equal(pc, qc)


def test_pow2_amax_element_keeps_at_least_half_the_range():
    rng = np.random.default_rng(53)
    x = rng.standard_normal((64, 128)).astype(np.float32)
    codes, s = Q.quantize(x, Q.ROWWISE, Q.ACT, pow2=True)
    amax_idx = np.argmax(np.abs(x), axis=1)
    top = e4m3.decode(codes[np.arange(64), amax_idx] & 0x7F)
    assert np.all(top >= 224) and np.all(top <= 448)  # S < 2 fl32(amax/448): amax / S > 224
