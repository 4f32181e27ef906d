"""Pins for the oracle's clipped surrogate (Eq. 1, Eq. 4, §2.1 clip semantics).

A hand-worked table, the unclipped special case r = 1 (loss reduces to the
TIS-weighted mean of -A), A = 0, the equality conventions, and the gradient
against a central finite difference in float64.
"""

import os

import numpy as np
import pytest

from oracle import surrogate as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_hand_worked_table():
    rows = []
    for line in open(os.path.join(GOLDEN, "surrogate_tiny.txt")):
        line = line.split("#")[0].strip()
        if line:
            rows.append([float(x) for x in line.split()[:6]])
    a = np.array(rows)
    r, adv, w, mask, term, clipped = (a[:, i] for i in range(6))
    out = S.clipped_surrogate(r, adv, mask, w, 0.8, 1.2)
    assert np.allclose(out["terms"], term, rtol=0, atol=1e-6)
    assert np.array_equal(out["clip_mask"] != 0, clipped != 0)
    assert abs(out["loss"] - 0.3 / 7) < 1e-6
    assert out["n_valid"] == 7 and out["clipped_pos"] == 2 and out["clipped_neg"] == 2
    # clip fractions by sign (§3): 2 of the 4 valid A>0 tokens, 2 of the 3 A<0
    # tokens, 4 of the 7 valid tokens
    assert out["clip_frac_pos"] == 2 / 4 and out["clip_frac_neg"] == 2 / 3 and out["clip_frac"] == 4 / 7


def test_unclipped_ratio_one():
    rng = np.random.default_rng(0)
    adv = rng.standard_normal(100).astype(np.float32)
    w = rng.uniform(0.5, 2, 100).astype(np.float32)
    mask = (rng.random(100) < 0.8).astype(np.uint8)
    out = S.clipped_surrogate(np.ones(100, np.float32), adv, mask, w, 0.8, 1.2)
    v = mask != 0
    assert np.isclose(out["loss"], -np.sum(w[v].astype(np.float64) * adv[v]) / v.sum(), rtol=1e-14)
    assert out["clipped_pos"] == 0 and out["clipped_neg"] == 0


def test_zero_advantage_and_empty_mask():
    out = S.clipped_surrogate(np.full(5, 3.0), np.zeros(5), np.ones(5), None, 0.8, 1.2)
    assert out["loss"] == 0 and np.all(out["grad"] == 0) and np.all(out["clip_mask"] == 0)
    out = S.clipped_surrogate(np.full(5, 3.0), np.ones(5), np.zeros(5), None, 0.8, 1.2)
    assert out["loss"] == 0 and out["n_valid"] == 0


@pytest.mark.parametrize("seed", range(5))
def test_gradient_finite_difference(seed):
    rng = np.random.default_rng(seed)
    T = 40
    logp_old = rng.normal(-3, 1, T)
    logp = logp_old + rng.normal(0, 0.3, T)
    adv = rng.standard_normal(T)
    w = rng.uniform(0.5, 2, T)
    mask = (rng.random(T) < 0.8).astype(np.uint8)
    lo, hi = 0.8, 1.2
    r = np.exp(logp - logp_old)
    # keep away from the kinks so the finite difference is clean
    near = (np.abs(r - lo) < 1e-3) | (np.abs(r - hi) < 1e-3)
    logp[near] += 0.01

    def loss(lp):
        rr = np.exp(lp - logp_old)
        lo64, hi64 = float(np.float32(lo)), float(np.float32(hi))
        t = -w * np.minimum(rr * adv, np.clip(rr, lo64, hi64) * adv)
        return np.sum(np.where(mask != 0, t, 0)) / max(1, mask.sum())

    r = np.exp(logp - logp_old)
    # gradient of the oracle, evaluated in float64 terms
    out = S.clipped_surrogate(r, adv, mask, w, lo, hi)
    h = 1e-7
    for t in range(T):
        e = np.zeros(T)
        e[t] = h
        fd = (loss(logp + e) - loss(logp - e)) / (2 * h)
        assert abs(fd - out["grad"][t]) < 5e-6 * max(1, abs(fd)), t


def test_absent_mask_means_all_valid():
    r = np.array([1.0, 1.5, 0.5], np.float32)
    a = np.array([1.0, 1.0, -1.0], np.float32)
    out = S.clipped_surrogate(r, a, None, None, 0.8, 1.2)
    ref = S.clipped_surrogate(r, a, np.ones(3, np.uint8), None, 0.8, 1.2)
    assert out["n_valid"] == 3 and out["loss"] == ref["loss"]


# ---- sequence-mean variant (GRPO's 1/|o_i| normalisation) -------------------

def _seq_inputs(rng, T, n_seq, equal=False):
    r = np.exp(rng.normal(0, 0.3, T)).astype(np.float32)
    A = rng.normal(0, 1, T).astype(np.float32)
    w = rng.uniform(0.5, 2.0, T).astype(np.float32)
    if equal:
        sid = np.repeat(np.arange(n_seq), T // n_seq)
        m = np.ones(T, np.uint8)
    else:
        sid = rng.integers(0, n_seq, T)
        m = (rng.random(T) < 0.8).astype(np.uint8)
    return r, A, w, m, sid


def test_seq_mean_equals_token_mean_for_equal_lengths():
    rng = np.random.default_rng(20)
    r, A, w, m, sid = _seq_inputs(rng, 120, 6, equal=True)
    tok = S.clipped_surrogate(r, A, m, w, 0.8, 1.2)
    seq = S.clipped_surrogate_seq_mean(r, A, m, w, 0.8, 1.2, sid, 6)
    assert abs(seq["loss"] - tok["loss"]) < 1e-12
    assert np.allclose(seq["grad"], tok["grad"], rtol=0, atol=1e-15)


def test_seq_mean_single_sequence_and_hand_case():
    rng = np.random.default_rng(21)
    r, A, w, m, _ = _seq_inputs(rng, 50, 1)
    tok = S.clipped_surrogate(r, A, m, w, 0.8, 1.2)
    seq = S.clipped_surrogate_seq_mean(r, A, m, w, 0.8, 1.2, np.zeros(50, int), 1)
    assert abs(seq["loss"] - tok["loss"]) < 1e-12
    # two sequences, lengths 1 and 3, unclipped ratios 1, A = 1 / 2 / 3 / 6:
    # terms -1 | -2, -3, -6 -> means -1 and -11/3 -> loss -(1 + 11/3)/2 = -7/3
    one = np.ones(4, np.float32)
    res = S.clipped_surrogate_seq_mean(one, np.float32([1, 2, 3, 6]), None, None, 0.8, 1.2,
                                       [0, 1, 1, 1], 3)  # sequence 2 has no tokens
    assert abs(res["loss"] - (-7.0 / 3.0)) < 1e-15 and res["n_seq_valid"] == 2
    assert np.allclose(res["grad"], [-1.0 / 2, -2.0 / 6, -3.0 / 6, -6.0 / 6], rtol=0, atol=1e-15)


def test_seq_mean_permutation_invariance_and_empty():
    rng = np.random.default_rng(22)
    r, A, w, m, sid = _seq_inputs(rng, 200, 17)
    a = S.clipped_surrogate_seq_mean(r, A, m, w, 0.8, 1.2, sid, 17)
    p = rng.permutation(200)
    b = S.clipped_surrogate_seq_mean(r[p], A[p], m[p], w[p], 0.8, 1.2, sid[p], 17)
    assert abs(a["loss"] - b["loss"]) < 1e-12
    assert np.allclose(a["grad"][p], b["grad"], rtol=0, atol=1e-15)
    e = S.clipped_surrogate_seq_mean(r, A, np.zeros(200, np.uint8), w, 0.8, 1.2, sid, 17)
    assert e["loss"] == 0.0 and e["n_seq_valid"] == 0 and not np.any(e["grad"])
    with pytest.raises(ValueError):
        S.clipped_surrogate_seq_mean(r, A, m, w, 0.8, 1.2, np.full(200, 17), 17)


def test_seq_mean_gradient_finite_difference():
    # the oracle's g_t against a central difference of the float64 loss as a
    # function of logp (r = exp(logp - logp_old)), away from the clip kinks
    rng = np.random.default_rng(23)
    T, n = 30, 4
    lp_old = rng.normal(-3, 1, T)
    lp = lp_old + rng.normal(0, 0.05, T)
    A = rng.normal(0, 1, T)
    sid = rng.integers(0, n, T)
    m = (rng.random(T) < 0.8).astype(np.uint8)
    lo, hi = 0.5, 2.0

    def loss(x):
        rr = np.exp(x - lp_old)
        term = -np.minimum(rr * A, np.clip(rr, lo, hi) * A) * (m != 0)
        cnt = np.bincount(sid, weights=(m != 0).astype(float), minlength=n)
        sums = np.bincount(sid, weights=term, minlength=n)
        keep = cnt > 0
        return np.sum(sums[keep] / cnt[keep]) / keep.sum()

    g = S.clipped_surrogate_seq_mean(np.exp(lp - lp_old), A, m, None, lo, hi, sid, n)["grad"]
    h = 1e-7
    for t in range(T):
        e = np.zeros(T)
        e[t] = h
        fd = (loss(lp + e) - loss(lp - e)) / (2 * h)
        assert abs(fd - g[t]) < 5e-6 * max(1.0, abs(fd)), t


# ---- sequence-level ratio clipping (one geometric-mean ratio per response) ---

def test_seq_level_hand_case():
    # sequence 0: d = ln 2, 0 -> s = sqrt 2 >= H with A > 0: clipped, term -H
    # sequence 1: d = 0, 0, 0 -> s = 1, A = -1: term +1, g = -A s / (n S) = 1/9
    # sequence 2: d = -ln 4 -> s = 1/4 <= L with A < 0: clipped, term -A L = 0.5 L
    lp = np.array([np.log(2), 0, 0, 0, 0, -np.log(4)], np.float32)
    out = S.seq_level_clipped_surrogate(lp, np.zeros(6, np.float32), [1.0, -1.0, -0.5], None,
                                        [0, 0, 1, 1, 1, 2], 3, 0.8, 1.2)
    L32, H32 = float(np.float32(0.8)), float(np.float32(1.2))
    assert np.allclose(out["seq_ratio"], [np.sqrt(2.0), 1.0, 0.25], rtol=1e-7, atol=0)
    assert list(out["seq_clip"]) == [S.CLIP_HI, 0, S.CLIP_LO]
    assert abs(out["loss"] - (-H32 + 1.0 + 0.5 * L32) / 3) < 1e-15
    assert np.allclose(out["grad"], [0, 0, 1 / 9, 1 / 9, 1 / 9, 0], rtol=0, atol=1e-15)
    assert out["n_seq_valid"] == 3 and out["clipped_pos"] == 1 and out["clipped_neg"] == 1
    # fractions over responses: 1 of 1 with A > 0, 1 of 2 with A < 0, 2 of 3
    assert out["clip_frac_pos"] == 1.0 and out["clip_frac_neg"] == 0.5 and out["clip_frac"] == 2 / 3


def test_seq_level_ratio_is_geometric_mean_of_token_ratios():
    # the literal definition (pi(y)/pi_old(y))^(1/|y|) with pi(y) the product of
    # the token probabilities, on short sequences where the products stay finite
    rng = np.random.default_rng(30)
    n_seq, T = 9, 60
    sid = rng.integers(0, n_seq, T)
    lp = rng.normal(-2, 0.7, T).astype(np.float32)
    lp_old = (lp + rng.normal(0, 0.2, T)).astype(np.float32)
    m = (rng.random(T) < 0.85).astype(np.uint8)
    out = S.seq_level_clipped_surrogate(lp, lp_old, np.ones(n_seq), m, sid, n_seq, 0.0, np.inf)
    for i in range(n_seq):
        sel = (sid == i) & (m != 0)
        if not sel.any():
            assert out["seq_ratio"][i] == 0 and out["seq_valid_tokens"][i] == 0
            continue
        d = (lp[sel] - lp_old[sel]).astype(np.float64)  # the float32 token log-ratios
        geo = np.prod(np.exp(d)) ** (1.0 / sel.sum())
        assert abs(out["seq_ratio"][i] - geo) < 1e-13 * geo, i


def test_seq_level_single_token_sequences_reduce_to_token_level():
    # one valid token per sequence: s_i is that token's ratio, S = n_valid, and
    # the loss, clip bits and gradient are the token-mean surrogate's
    rng = np.random.default_rng(31)
    T = 300
    d = rng.normal(0, 0.3, T).astype(np.float32)
    lp_old = rng.normal(-3, 1, T).astype(np.float32)
    lp = (lp_old + d).astype(np.float32)
    A = rng.normal(0, 1, T).astype(np.float32)
    A[::17] = 0
    out = S.seq_level_clipped_surrogate(lp, lp_old, A, None, np.arange(T), T, 0.8, 1.2)
    r = np.float32(np.exp((lp - lp_old).astype(np.float64)))
    tok = S.clipped_surrogate(r, A, None, None, 0.8, 1.2)
    assert abs(out["loss"] - tok["loss"]) < 1e-14
    assert np.array_equal(out["seq_clip"], tok["clip_mask"])
    assert np.allclose(out["grad"], tok["grad"], rtol=1e-15, atol=0)
    assert (out["clipped_pos"], out["clipped_neg"]) == (tok["clipped_pos"], tok["clipped_neg"])


def test_seq_level_unclipped_and_invariances():
    rng = np.random.default_rng(32)
    T, n = 400, 23
    sid = rng.integers(0, n, T)
    lp_old = rng.normal(-3, 1, T).astype(np.float32)
    lp = (lp_old + rng.normal(0, 0.5, T)).astype(np.float32)
    A = rng.normal(0, 1, n).astype(np.float32)
    m = (rng.random(T) < 0.7).astype(np.uint8)
    # bounds that clip nothing: loss = -(1/S) sum_i A_i s_i
    free = S.seq_level_clipped_surrogate(lp, lp_old, A, m, sid, n, 0.0, np.inf)
    live = free["seq_valid_tokens"] > 0
    s32 = free["seq_ratio32"].astype(np.float64)
    assert abs(free["loss"] - (-np.sum(A[live] * s32[live]) / live.sum())) < 1e-14
    assert free["clipped_pos"] == 0 and free["clipped_neg"] == 0
    # token order and sequence labels do not matter
    a = S.seq_level_clipped_surrogate(lp, lp_old, A, m, sid, n, 0.8, 1.2)
    p = rng.permutation(T)
    relabel = rng.permutation(n)
    b = S.seq_level_clipped_surrogate(lp[p], lp_old[p], A[np.argsort(relabel)], m[p], relabel[sid[p]],
                                      n, 0.8, 1.2)
    assert abs(a["loss"] - b["loss"]) < 1e-14
    assert np.array_equal(a["grad"][p], b["grad"])
    assert np.array_equal(a["seq_clip"], b["seq_clip"][relabel])


def test_seq_level_empty_and_bad_input():
    lp = np.zeros(8, np.float32)
    out = S.seq_level_clipped_surrogate(lp, lp, np.ones(3), np.zeros(8, np.uint8), np.zeros(8, int), 3,
                                        0.8, 1.2)
    assert out["loss"] == 0 and out["n_seq_valid"] == 0 and not out["grad"].any()
    with pytest.raises(ValueError):
        S.seq_level_clipped_surrogate(lp, lp, np.ones(3), None, np.full(8, 3), 3, 0.8, 1.2)
    big = lp.copy()
    big[2] = 200.0
    with pytest.raises(ValueError):
        S.seq_level_clipped_surrogate(big, lp, np.ones(3), None, np.zeros(8, int), 3, 0.8, 1.2)
    # a masked token may hold anything
    m = np.ones(8, np.uint8)
    m[2] = 0
    S.seq_level_clipped_surrogate(big, lp, np.ones(3), m, np.zeros(8, int), 3, 0.8, 1.2)


def test_seq_level_gradient_finite_difference():
    rng = np.random.default_rng(33)
    T, n = 40, 5
    sid = rng.integers(0, n, T)
    lp_old = rng.normal(-3, 1, T)
    lp = lp_old + rng.normal(0, 0.2, T)
    A = rng.normal(0, 1, n)
    m = (rng.random(T) < 0.8).astype(np.uint8)
    lo, hi = 0.9, 1.1

    def loss(x):
        v = m != 0
        cnt = np.bincount(sid[v], minlength=n)
        mu = np.bincount(sid[v], weights=(x - lp_old)[v], minlength=n)
        keep = cnt > 0
        s = np.exp(mu[keep] / cnt[keep])
        a = A[keep]
        return np.sum(-np.minimum(s * a, np.clip(s, lo, hi) * a)) / keep.sum()

    g = S.seq_level_clipped_surrogate(lp, lp_old, A, m, sid, n, lo, hi)["grad"]
    h = 1e-6
    for t in range(T):
        e = np.zeros(T)
        e[t] = h
        fd = (loss(lp + e) - loss(lp - e)) / (2 * h)
        assert abs(fd - g[t]) < 1e-5 * max(1.0, abs(fd)), t
