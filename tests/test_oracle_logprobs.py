"""Pins for the oracle's FP8 logits / log-prob / dlogits (§2.1, Eq. 3).

Closed forms (W = 0, V = 1), one-hot weight rows (catches a transposed or
mis-indexed operand), scale-exchange invariance between the two operands'
block scales (catches a dropped or misplaced scale), SciPy's log_softmax, the
normalisation of the softmax, and a finite-difference check of dlogits.

The BF16 shadow-pass scorer (§4) is pinned by its closed forms, one-hot rows,
and by agreement with the (separately pinned) FP8 path on operands that E4M3
represents exactly with scale 1, where quantisation changes nothing.
"""

import numpy as np
import pytest
import scipy.special

from oracle import e4m3
from oracle import logprobs as L
from oracle import quantize as Q


def _codes(rng, shape):
    c = rng.integers(0, 256, size=shape).astype(np.uint8)
    c[(c == 0x7F) | (c == 0xFF)] = 0x38
    return c


@pytest.mark.parametrize("gran", [Q.TENSOR, Q.ROWWISE, Q.BLOCK])
def test_zero_weight_gives_uniform(gran):
    rng = np.random.default_rng(0)
    T, H, V = 5, 256, 37
    hc = _codes(rng, (T, H))
    hs = {Q.TENSOR: np.float32([0.5]), Q.ROWWISE: np.full(T, 0.25, np.float32),
          Q.BLOCK: np.full((T, 2), 0.125, np.float32)}[gran]
    wc = np.zeros((V, H), np.uint8)
    ws = {Q.TENSOR: np.float32([1.0]), Q.ROWWISE: np.ones(V, np.float32),
          Q.BLOCK: np.ones((1, 2), np.float32)}[gran]
    y = rng.integers(0, V, T)
    logp, lse = L.token_logprobs(hc, hs, wc, ws, gran, y)
    assert np.allclose(logp, -np.log(V), rtol=0, atol=1e-14)


def test_single_word_vocab():
    rng = np.random.default_rng(1)
    hc = _codes(rng, (4, 128))
    wc = _codes(rng, (1, 128))
    logp, _ = L.token_logprobs(hc, np.float32([0.01]), wc, np.float32([0.02]), Q.TENSOR, [0, 0, 0, 0])
    assert np.all(logp == 0.0)


def test_one_hot_rows_pick_dequantised_hidden_entries():
    rng = np.random.default_rng(2)
    T, H, V = 6, 256, 9
    hc = _codes(rng, (T, H))
    hs = rng.uniform(0.01, 2, size=(T, H // 128)).astype(np.float32)
    cols = rng.integers(0, H, V)
    wc = np.zeros((V, H), np.uint8)
    wc[np.arange(V), cols] = 0x38  # code for 1.0
    ws = np.ones((1, H // 128), np.float32)
    z = L.logits(hc, hs, wc, ws, Q.BLOCK)
    expect = e4m3.decode(hc)[:, cols] * hs[:, cols // 128]
    assert np.array_equal(z, expect)


def test_block_scale_exchange_invariance():
    rng = np.random.default_rng(3)
    T, H, V = 7, 384, 200
    hc, wc = _codes(rng, (T, H)), _codes(rng, (V, H))
    hs = rng.uniform(0.01, 1, size=(T, 3)).astype(np.float32)
    ws = rng.uniform(0.01, 1, size=(2, 3)).astype(np.float32)
    z0 = L.logits(hc, hs, wc, ws, Q.BLOCK)
    hs2, ws2 = hs.copy(), ws.copy()
    hs2[:, 1] *= 4
    ws2[:, 1] /= 4
    assert np.allclose(L.logits(hc, hs2, wc, ws2, Q.BLOCK), z0, rtol=1e-13, atol=1e-13)
    ws3 = ws.copy()
    ws3[:, 1] *= 2  # changing one scale must change the result
    assert not np.allclose(L.logits(hc, hs, wc, ws3, Q.BLOCK), z0)
    # equal block scales per row reduce block mode to row mode
    hs_row = rng.uniform(0.01, 1, size=T).astype(np.float32)
    ws_row = np.full(V, 0.5, np.float32)
    zr = L.logits(hc, hs_row, wc, ws_row, Q.ROWWISE)
    zb = L.logits(hc, np.repeat(hs_row[:, None], 3, 1), wc, np.full((2, 3), 0.5, np.float32), Q.BLOCK)
    assert np.allclose(zr, zb, rtol=1e-14, atol=1e-14)


def test_log_softmax_matches_scipy_and_normalises():
    rng = np.random.default_rng(4)
    z = rng.standard_normal((8, 1000)) * 5
    y = rng.integers(0, 1000, 8)
    logp, lse = L.log_softmax_gather(z, y)
    ref = scipy.special.log_softmax(z, axis=1)[np.arange(8), y]
    assert np.allclose(logp, ref, rtol=0, atol=1e-12)
    assert np.allclose(lse, scipy.special.logsumexp(z, axis=1), rtol=0, atol=1e-12)
    all_logp = np.stack([L.log_softmax_gather(z, np.full(8, v))[0] for v in range(1000)], 1)
    assert np.allclose(np.exp(all_logp).sum(1), 1.0, atol=1e-12)
    with pytest.raises(ValueError):
        L.log_softmax_gather(z, np.full(8, 1000))


def test_dlogits_finite_difference():
    rng = np.random.default_rng(5)
    T, V = 3, 11
    z = rng.standard_normal((T, V))
    y = rng.integers(0, V, T)
    g = rng.standard_normal(T)

    def f(zz):
        return float(np.sum(g * L.log_softmax_gather(zz, y)[0]))

    _, lse = L.log_softmax_gather(z, y)
    d = L.dlogits(z, y, lse, g)
    h = 1e-6
    for t in range(T):
        for v in range(V):
            zp, zm = z.copy(), z.copy()
            zp[t, v] += h
            zm[t, v] -= h
            assert abs((f(zp) - f(zm)) / (2 * h) - d[t, v]) < 1e-8
    assert np.allclose(d.sum(1), 0.0, atol=1e-14)


def test_ratio_identity():
    lp = np.random.default_rng(6).standard_normal(10)
    assert np.all(L.importance_ratios(lp, lp) == 1.0)


def _bf16_values(rng, shape, std):
    """Random float32 values that are exactly representable in bf16."""
    x = (rng.standard_normal(shape) * std).astype(np.float32)
    return (x.view(np.uint32) & np.uint32(0xFFFF0000)).view(np.float32)


def test_bf16_zero_weight_and_single_word():
    rng = np.random.default_rng(10)
    h = _bf16_values(rng, (6, 64), 1.0)
    lp, lse = L.bf16_token_logprobs(h, np.zeros((29, 64), np.float32), rng.integers(0, 29, 6))
    assert np.allclose(lp, -np.log(29), rtol=0, atol=1e-14)
    assert np.allclose(lse, np.log(29), rtol=0, atol=1e-14)
    lp1, _ = L.bf16_token_logprobs(h, _bf16_values(rng, (1, 64), 0.02), np.zeros(6, np.int64))
    assert np.all(lp1 == 0.0)


def test_bf16_one_hot_rows_pick_hidden_entries():
    rng = np.random.default_rng(11)
    T, H, V = 5, 96, 13
    h = _bf16_values(rng, (T, H), 1.0)
    cols = rng.integers(0, H, V)
    W = np.zeros((V, H), np.float32)
    W[np.arange(V), cols] = 1.0
    assert np.array_equal(L.bf16_logits(h, W), h[:, cols].astype(np.float64))
    rows = np.array([4, 1])
    assert np.array_equal(L.bf16_logits(h, W, rows), h[rows][:, cols].astype(np.float64))


def test_bf16_path_equals_fp8_path_on_exact_e4m3_operands():
    # every finite E4M3 value is a bf16 value; with one entry of +-448 per
    # tensor the per-tensor scale is exactly 1 and the codes decode to the
    # inputs, so both scorers see identical operands
    rng = np.random.default_rng(12)
    T, H, V = 7, 128, 50
    finite = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], np.uint8)
    vals = e4m3.decode(finite).astype(np.float32)
    h = rng.choice(vals, size=(T, H)).astype(np.float32)
    W = rng.choice(vals, size=(V, H)).astype(np.float32)
    h[0, 0] = 448.0
    W[3, 5] = -448.0
    hq, hs = Q.quantize(h, Q.TENSOR, Q.ACT)
    wq, ws = Q.quantize(W, Q.TENSOR, Q.WEIGHT)
    assert hs[0] == 1.0 and ws[0] == 1.0
    y = rng.integers(0, V, T)
    lp8, lse8 = L.token_logprobs(hq, hs, wq, ws, Q.TENSOR, y)
    lpb, lseb = L.bf16_token_logprobs(h, W, y)
    assert np.array_equal(lp8, lpb) and np.array_equal(lse8, lseb)
    # and a perturbation that E4M3 cannot represent separates them
    h2 = h.copy()
    h2[1, 1] = np.float32(1.0078125)  # 1 + 2^-7: bf16-exact, not E4M3-exact
    hq2, hs2 = Q.quantize(h2, Q.TENSOR, Q.ACT)
    assert not np.array_equal(L.token_logprobs(hq2, hs2, wq, ws, Q.TENSOR, y)[0],
                              L.bf16_token_logprobs(h2, W, y)[0])


# ---- backward through the lm_head -------------------------------------------

def _exact_operands(rng, shape, amax):
    """Values e/512 for finite E4M3 values e, with one entry +-448/512: the
    per-tensor scale fl32(amax/448) is exactly 2^-9 and every value divided by
    it is an E4M3 value, so the codes decode to the inputs exactly."""
    finite = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], np.uint8)
    vals = e4m3.decode(finite).astype(np.float64) / 512
    x = rng.choice(vals, size=shape)
    x.flat[0] = amax
    return x


def test_lm_head_backward_finite_difference():
    # L(h, W) = sum_t g_t log_softmax(h W^T)[t, y_t], written out in float64
    # from the operands; at an on-grid point (quantisation changes nothing)
    # its gradient is the oracle's dh, dW
    rng = np.random.default_rng(40)
    T, H, V = 5, 16, 11
    h = _exact_operands(rng, (T, H), 448.0 / 512)
    W = _exact_operands(rng, (V, H), -448.0 / 512)
    hq, hs = Q.quantize(h.astype(np.float32), Q.TENSOR, Q.ACT)
    wq, ws = Q.quantize(W.astype(np.float32), Q.TENSOR, Q.WEIGHT)
    assert hs[0] == 2.0 ** -9 and ws[0] == 2.0 ** -9
    assert np.array_equal(Q.dequantize(hq, hs, Q.TENSOR, Q.ACT), h)
    assert np.array_equal(Q.dequantize(wq, ws, Q.TENSOR, Q.WEIGHT), W)
    y = rng.integers(0, V, T)
    g = rng.normal(0, 1, T)

    def loss(hh, WW):
        z = hh @ WW.T
        m = z.max(axis=1, keepdims=True)
        lse = (m + np.log(np.exp(z - m).sum(axis=1, keepdims=True)))[:, 0]
        return float(np.sum(g * (z[np.arange(T), y] - lse)))

    out = L.lm_head_backward(hq, hs, wq, ws, Q.TENSOR, y, g, h, W)
    eps = 1e-6
    for (t, k) in [(0, 1), (2, 5), (4, 15), (1, 0)]:
        e = np.zeros_like(h)
        e[t, k] = eps
        fd = (loss(h + e, W) - loss(h - e, W)) / (2 * eps)
        assert abs(fd - out["dh"][t, k]) < 1e-7 * max(1.0, abs(fd)), (t, k)
    for (v, k) in [(0, 0), (3, 7), (10, 15), (6, 2)]:
        e = np.zeros_like(W)
        e[v, k] = eps
        fd = (loss(h, W + e) - loss(h, W - e)) / (2 * eps)
        assert abs(fd - out["dW"][v, k]) < 1e-7 * max(1.0, abs(fd)), (v, k)


def test_lm_head_backward_uniform_softmax_closed_form():
    # all weight rows equal: the softmax is uniform, dh = 0 and
    # dW[v] = sum_{t: y_t = v} g_t h_t - (1/V) sum_t g_t h_t
    rng = np.random.default_rng(41)
    T, H, V = 9, 32, 7
    h = rng.normal(0, 1, (T, H)).astype(np.float32)
    W = np.tile(rng.normal(0, 0.1, (1, H)), (V, 1)).astype(np.float32)
    hq, hs = Q.quantize(h, Q.ROWWISE, Q.ACT)
    wq, ws = Q.quantize(W, Q.ROWWISE, Q.WEIGHT)
    y = rng.integers(0, V, T)
    g = rng.normal(0, 1, T)
    out = L.lm_head_backward(hq, hs, wq, ws, Q.ROWWISE, y, g, h, W)
    assert np.abs(out["dh"]).max() < 1e-12
    gh = g[:, None] * h.astype(np.float64)
    want = np.zeros((V, H))
    for t in range(T):
        want[y[t]] += gh[t]
    want -= gh.sum(axis=0) / V
    assert np.allclose(out["dW"], want, rtol=0, atol=1e-12)


@pytest.mark.parametrize("gran", [Q.TENSOR, Q.ROWWISE, Q.BLOCK])
def test_lm_head_backward_invariants(gran):
    rng = np.random.default_rng(42 + gran)
    T, H, V = 6, 256, 300
    h = rng.normal(0, 1, (T, H)).astype(np.float32)
    W = rng.normal(0, 0.05, (V, H)).astype(np.float32)
    hq, hs = Q.quantize(h, gran, Q.ACT)
    wq, ws = Q.quantize(W, gran, Q.WEIGHT)
    y = rng.integers(0, V, T)
    g = rng.normal(0, 1, T)
    out = L.lm_head_backward(hq, hs, wq, ws, gran, y, g, h, W)
    # every row of P sums to g_t (1 - 1) = 0, so the columns of dW sum to 0
    assert np.abs(out["P"].sum(axis=1)).max() < 1e-12
    assert np.abs(out["dW"].sum(axis=0)).max() < 1e-10 * np.abs(out["dW"]).sum(axis=0).max()
    # g = 0 gives nothing; rows= gives the same dh rows
    z = L.lm_head_backward(hq, hs, wq, ws, gran, y, np.zeros(T), h, W)
    assert not z["dh"].any() and not z["dW"].any()
    part = L.lm_head_backward(hq, hs, wq, ws, gran, y, g, h, W, rows=[4, 1])
    assert np.allclose(part["dh"], out["dh"][[4, 1]], rtol=0, atol=1e-13 * np.abs(out["dh"]).max())
    assert "dW" not in part


# ---- FP8 backward (both contractions on E4M3 operands) -----------------------

def test_fp8_backward_equals_exact_backward_when_quantisation_is_exact():
    # 128 identical tokens, V = 2: every row of P is (a, -a) or (-a, a), so each
    # 1x128 block of P and each 128 x 128 block of P^T holds one magnitude and
    # encodes to +-448 exactly; W and h sit on the E4M3 grid with amax 448 2^-9,
    # so their 128 x 128 quantisation is exact too.  The FP8 backward must then
    # equal the exact one up to the float32 rounding of P and of its scales.
    rng = np.random.default_rng(71)
    T, H, V = 128, 128, 2
    h_row = _exact_operands(rng, (1, H), 448.0 / 512)
    h = np.repeat(h_row, T, axis=0)
    W = _exact_operands(rng, (V, H), -448.0 / 512)
    hq, hs = Q.quantize(h.astype(np.float32), Q.BLOCK, Q.ACT)
    wq, ws = Q.quantize(W.astype(np.float32), Q.BLOCK, Q.WEIGHT)
    y = np.zeros(T, np.int64)
    g = np.full(T, 0.37)
    ref = L.lm_head_backward(hq, hs, wq, ws, Q.BLOCK, y, g, h, W)
    out = L.lm_head_backward_fp8(hq, hs, wq, ws, Q.BLOCK, y, g, h, W)
    assert np.array_equal(out["Wt_hat"], W.T) and np.array_equal(out["ht_hat"], h.T)
    assert np.all(np.abs(out["p_codes"][:, :V]) != 0)
    for k in ("dh", "dW"):
        bound = 2.0 ** -22 * (np.abs(ref["P"]) @ np.abs(W) if k == "dh" else np.abs(ref["P"]).T @ np.abs(h))
        assert np.all(np.abs(out[k] - ref[k]) <= bound + 1e-300), k
    assert np.max(np.abs(ref["dh"])) > 0 and np.max(np.abs(ref["dW"])) > 0


def _e4m3_abs_err_bound(x, scale_of):
    # |Q(x) - x| <= max(2^-4 |x|, 2^-10 S): half a step of the 3-bit mantissa
    # in the normal range, half the subnormal step 2^-9 S below it
    return np.maximum(2.0 ** -4 * np.abs(x), 2.0 ** -10 * scale_of)


@pytest.mark.parametrize("gran,pow2", [(Q.TENSOR, False), (Q.ROWWISE, False), (Q.BLOCK, False),
                                       (Q.BLOCK, True)])
def test_fp8_backward_within_quantisation_error_of_exact_backward(gran, pow2):
    # dh = sum_v P W and dW = sum_t P^T h with every operand quantised: the
    # difference to the exact contraction is bounded term by term by the E4M3
    # rounding of both factors.  A dropped or misplaced scale, a transposed
    # operand or a wrong block index breaks the bound by orders of magnitude.
    # Power-of-two scales keep |x / S| <= 448, so the same bound holds.
    rng = np.random.default_rng(72 + gran + 7 * pow2)
    T, H, V = 130, 256, 300
    h = rng.normal(0, 1, (T, H)).astype(np.float32)
    W = (rng.normal(0, 0.05, (V, H))).astype(np.float32)
    hq, hs = Q.quantize(h, gran, Q.ACT, pow2=pow2)
    wq, ws = Q.quantize(W, gran, Q.WEIGHT, pow2=pow2)
    y = rng.integers(0, V, T)
    g = rng.normal(0, 1, T) / T
    ref = L.lm_head_backward(hq, hs, wq, ws, gran, y, g, h, W)
    out = L.lm_head_backward_fp8(hq, hs, wq, ws, gran, y, g, h, W, pow2=pow2)
    P = out["P"].astype(np.float64)
    # per-element scales of each quantised operand
    sp = np.repeat(out["p_scales"], 128, axis=1)[:, :V]
    spt = np.repeat(np.repeat(out["pt_scales"], 128, axis=0), 128, axis=1)[:V, :T]
    swt = np.repeat(np.repeat(out["wt_scales"], 128, axis=0), 128, axis=1)[:H, :V]
    sht = np.repeat(np.repeat(out["ht_scales"], 128, axis=0), 128, axis=1)[:H, :T]
    ep, ept = _e4m3_abs_err_bound(P, sp), _e4m3_abs_err_bound(P.T, spt)
    ew, eh = _e4m3_abs_err_bound(W.T, swt), _e4m3_abs_err_bound(h.T, sht)
    assert np.all(np.abs(out["P_hat"] - P) <= ep) and np.all(np.abs(out["Wt_hat"] - W.T) <= ew)
    assert np.all(np.abs(out["Pt_hat"] - P.T) <= ept) and np.all(np.abs(out["ht_hat"] - h.T) <= eh)
    # the exact backward of the oracle, from P in float32 (the quantised one's input)
    dh_exact = P @ W.astype(np.float64)
    dW_exact = P.T @ h.astype(np.float64)
    assert np.allclose(dh_exact, ref["dh"], rtol=0, atol=1e-6 * np.max(np.abs(ref["dh"])))
    bound_dh = ep @ np.abs(W.astype(np.float64)) + (np.abs(P) + ep) @ ew.T
    bound_dW = ept @ np.abs(h.astype(np.float64)) + (np.abs(P.T) + ept) @ eh.T
    assert np.all(np.abs(out["dh"] - dh_exact) <= bound_dh * (1 + 1e-9))
    assert np.all(np.abs(out["dW"] - dW_exact) <= bound_dW * (1 + 1e-9))
    # and quantisation did change something (the check is not vacuous)
    assert np.max(np.abs(out["dh"] - dh_exact)) > 0


def test_fp8_backward_zero_gradient():
    rng = np.random.default_rng(73)
    T, H, V = 9, 128, 20
    h = rng.normal(0, 1, (T, H)).astype(np.float32)
    W = rng.normal(0, 0.05, (V, H)).astype(np.float32)
    hq, hs = Q.quantize(h, Q.BLOCK, Q.ACT)
    wq, ws = Q.quantize(W, Q.BLOCK, Q.WEIGHT)
    out = L.lm_head_backward_fp8(hq, hs, wq, ws, Q.BLOCK, rng.integers(0, V, T), np.zeros(T), h, W)
    assert not np.any(out["dh"]) and not np.any(out["dW"])
    # every block of P is zero: scale 1, codes +-0 (g * -p is -0.0)
    assert np.all(out["p_scales"] == 1.0) and np.all((out["p_codes"] & 0x7F) == 0)
    assert not np.any(out["P_hat"]) and not np.any(out["Pt_hat"])


def _is_pow2(s):
    m, _ = np.frexp(np.asarray(s, np.float64))
    return np.all(m == 0.5)


def test_fp8_backward_pow2_scales_by_brute_force():
    # The UE8M0 variant's backward: each operand's scale, found block by block
    # with Python loops over the unquantised operand, is the smallest power of
    # two S with amax / 448 <= S (S = 1 for a zero block), raised to 2^-127
    # where it falls below E8M0's range; the codes are RNE(x / S).  Row 0 has
    # g = 1e-41, so its P underflows far below 448 * 2^-127 and takes the floor.
    rng = np.random.default_rng(74)
    T, H, V = 130, 256, 200
    h = rng.normal(0, 1, (T, H)).astype(np.float32)
    W = rng.normal(0, 0.05, (V, H)).astype(np.float32)
    hq, hs = Q.quantize(h, Q.BLOCK, Q.ACT, pow2=True)
    wq, ws = Q.quantize(W, Q.BLOCK, Q.WEIGHT, pow2=True)
    y = rng.integers(0, V, T)
    g = rng.normal(0, 1, T) / T
    g[0] = 1e-41
    g[5] = 0.0
    out = L.lm_head_backward_fp8(hq, hs, wq, ws, Q.BLOCK, y, g, h, W, pow2=True)
    P = out["P"].astype(np.float64)

    def expected_scale(block):
        amax = float(np.max(np.abs(block))) if block.size else 0.0
        if amax == 0.0:
            return 1.0
        t = float(np.float32(np.float32(amax) / np.float32(448.0)))
        s = 2.0 ** -149
        while s < t:
            s *= 2.0
        return max(s, 2.0 ** -127)

    for t in range(T):
        for b in range(out["p_scales"].shape[1]):
            blk = P[t, 128 * b:128 * b + 128]
            assert out["p_scales"][t, b] == expected_scale(blk), (t, b)
    for vb in range(out["pt_scales"].shape[0]):
        for tb in range(out["pt_scales"].shape[1]):
            blk = P.T[128 * vb:128 * vb + 128, 128 * tb:128 * tb + 128]
            assert out["pt_scales"][vb, tb] == expected_scale(blk), (vb, tb)
    for hb in range(out["wt_scales"].shape[0]):
        for vb in range(out["wt_scales"].shape[1]):
            assert out["wt_scales"][hb, vb] == expected_scale(W.T[128 * hb:128 * hb + 128, 128 * vb:128 * vb + 128])
    assert out["p_scales"][0, y[0] // 128] == 2.0 ** -127 and P[0, y[0]] != 0
    assert np.all(out["p_scales"][5] == 1.0)
    for k in ("p_scales", "pt_scales", "wt_scales", "ht_scales"):
        assert _is_pow2(out[k]) and np.all(out[k] >= 2.0 ** -127), k
    # codes: RNE(x / S) with x / S exact (S a power of two)
    sp = np.repeat(out["p_scales"], 128, axis=1)[:, :V]
    q = (P / sp).astype(np.float32)
    assert np.array_equal(out["p_codes"][:, :V], e4m3.encode(q))
    assert np.array_equal(out["P_hat"], e4m3.decode(e4m3.encode(q)) * sp)
