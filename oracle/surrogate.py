"""Clipped PPO surrogate with TIS weights (Eq. 1, Eq. 4, §2.1) -- oracle side.

Test infrastructure only (see ``oracle/__init__.py``).

Eq. 1 / Eq. 4 per token, with calibrated bounds [L, H] in place of
[1 - eps, 1 + eps] (§4):

    l_t = -w_t * min(r_t A_t, clip(r_t, L, H) A_t),   clip(r, L, H) = min(max(r, L), H)

Clip semantics (§2.1): a token's gradient is zeroed when A_t > 0 and r_t >= H,
or A_t < 0 and r_t <= L -- these are the "clipped" tokens counted in the clip
fractions.

Readings:
* Aggregation is the token mean over valid tokens: loss = sum_{mask} l_t /
  sum mask (the DAPO token-level loss, used for GRPO as well).  sum mask = 0
  gives loss 0.
* The gradient returned is g_t = dloss / dlogp_t, with r_t = exp(logp_t -
  logp_old_t) so dr/dlogp = r: g_t = -w_t A_t r_t / sum mask on unclipped valid
  tokens and 0 elsewhere.
* w_t = 1 when no TIS weights are given.
* Everything here is float64.

Sequence-mean variant (GRPO's original normalisation, §2.1: the objective
averages each response's token terms, 1/|o_i| sum_t, then the responses):

    loss = (1/S) sum_{i : n_i > 0} (1/n_i) sum_{t in i, valid} l_t

with n_i the valid tokens of sequence i and S the sequences that have any;
g_t = -w_t A_t r_t / (S n_i) on unclipped valid tokens.  A sequence is the
set of tokens with the same id (they need not be contiguous).

Sequence-level ratio clipping (the GSPO-style trust region over whole
responses that the related-work discussion names, with extending calibration
to it left open): each response gets one ratio, the length-normalised
sequence likelihood ratio

    s_i = (pi(y_i) / pi_old(y_i))^(1/n_i) = exp((1/n_i) sum_{t in i, valid} d_t),
    d_t = logp_t - logp_old_t  (the float32 log of the token ratio),

i.e. the geometric mean of its token ratios, and one advantage A_i; the
clipped term, the clip rule (A_i > 0 and s_i >= H, or A_i < 0 and s_i <= L,
compared in float32 with s_i rounded to float32) and the aggregation over
responses follow the token-level definitions with s_i in place of r_t:

    loss = (1/S) sum_{i : n_i > 0} -A_i min(s_i, H)   (A_i >= 0)
                                   -A_i max(s_i, L)   (A_i < 0)
    g_t  = dloss/dlogp_t = -A_i s_i / (n_i S)  for valid t of unclipped i, else 0

(ds_i/dlogp_t = s_i / n_i).  A token log-ratio outside [-128, 128] (the
float32 token ratio would over- or underflow) or not finite is bad input.
"""

import numpy as np

CLIP_HI = 1  # bit set in the clip mask: A > 0 and r >= H
CLIP_LO = 2  # bit set in the clip mask: A < 0 and r <= L


def _valid(mask, n):
    """Valid-token mask; no mask means every token is valid."""
    return np.ones(n, bool) if mask is None else np.asarray(mask) != 0


def clip_mask(r, adv, mask, lo, hi):
    """Per-token clip bits, compared in float32 as the inputs are float32."""
    r = np.asarray(r, np.float32)
    adv = np.asarray(adv, np.float32)
    valid = _valid(mask, r.size)
    up = valid & (adv > 0) & (r >= np.float32(hi))
    dn = valid & (adv < 0) & (r <= np.float32(lo))
    return (up * CLIP_HI + dn * CLIP_LO).astype(np.uint8)


def clipped_surrogate(r, adv, mask, w, lo, hi):
    """Token-mean clipped surrogate loss, per-token terms, grad and counts."""
    r32 = np.asarray(r, np.float32)
    a32 = np.asarray(adv, np.float32)
    valid = _valid(mask, r32.size)
    r64 = r32.astype(np.float64)
    a64 = a32.astype(np.float64)
    w64 = np.ones_like(r64) if w is None else np.asarray(w, np.float32).astype(np.float64)
    lo64, hi64 = float(np.float32(lo)), float(np.float32(hi))
    clipped_r = np.minimum(np.maximum(r64, lo64), hi64)
    term = -w64 * np.minimum(r64 * a64, clipped_r * a64)
    term = np.where(valid, term, 0.0)
    n_valid = int(valid.sum())
    cm = clip_mask(r32, a32, valid, lo, hi)
    clipped = cm != 0
    loss_sum = float(np.sum(term))
    loss = loss_sum / n_valid if n_valid else 0.0
    grad = np.where(valid & ~clipped, -w64 * a64 * r64, 0.0)
    grad = grad / n_valid if n_valid else np.zeros_like(grad)
    n_pos = int(np.sum(valid & (a32 > 0)))
    n_neg = int(np.sum(valid & (a32 < 0)))
    c_pos = int(np.sum((cm & CLIP_HI) != 0))
    c_neg = int(np.sum((cm & CLIP_LO) != 0))
    return {
        "loss": loss, "loss_sum": loss_sum, "terms": term, "grad": grad,
        "clip_mask": cm, "n_valid": n_valid, "n_pos": n_pos, "n_neg": n_neg,
        "clipped_pos": c_pos, "clipped_neg": c_neg,
        "clip_frac_pos": c_pos / n_pos if n_pos else 0.0,
        "clip_frac_neg": c_neg / n_neg if n_neg else 0.0,
        "clip_frac": (c_pos + c_neg) / n_valid if n_valid else 0.0,
    }


def clipped_surrogate_seq_mean(r, adv, mask, w, lo, hi, seq_id, n_seq):
    """Sequence-mean of per-sequence token means of the clipped surrogate.

    Explicit per-sequence loop: the token terms, clip bits and counts are those
    of ``clipped_surrogate``; only the normalisation differs."""
    base = clipped_surrogate(r, adv, mask, w, lo, hi)
    r64 = np.asarray(r, np.float32).astype(np.float64)
    a64 = np.asarray(adv, np.float32).astype(np.float64)
    w64 = np.ones_like(r64) if w is None else np.asarray(w, np.float32).astype(np.float64)
    valid = _valid(mask, r64.size)
    sid = np.asarray(seq_id, np.int64)
    if np.any(sid < 0) or np.any(sid >= n_seq):
        raise ValueError("sequence id outside [0, n_seq)")
    clipped = base["clip_mask"] != 0
    n_i = np.zeros(n_seq, np.int64)
    for t in range(r64.size):
        if valid[t]:
            n_i[sid[t]] += 1
    S = int(np.sum(n_i > 0))
    seq_sums = np.zeros(n_seq)
    for t in range(r64.size):
        if valid[t]:
            seq_sums[sid[t]] += base["terms"][t]
    loss_sum = float(sum(seq_sums[i] / n_i[i] for i in range(n_seq) if n_i[i] > 0))
    grad = np.zeros_like(r64)
    for t in range(r64.size):
        if valid[t] and not clipped[t]:
            grad[t] = -w64[t] * a64[t] * r64[t] / (S * n_i[sid[t]])
    out = dict(base)
    out.update({"loss": loss_sum / S if S else 0.0, "loss_sum": loss_sum, "grad": grad,
                "n_seq_valid": S, "seq_valid_tokens": n_i})
    return out


D_MAX = 128.0  # largest |logp - logp_old| a valid token may have


def seq_level_clipped_surrogate(logp, logp_old, adv_seq, mask, seq_id, n_seq, lo, hi):
    """Sequence-level clipped surrogate: one ratio per response, the geometric
    mean of its token ratios, clipped like a token ratio.  Explicit loops over
    tokens and sequences; float64 throughout except the float32 token
    log-ratio and the float32 sequence ratio that the clip rule compares."""
    d32 = np.asarray(logp, np.float32) - np.asarray(logp_old, np.float32)  # float32 difference
    a_seq = np.asarray(adv_seq, np.float32).astype(np.float64)
    T = d32.size
    valid = _valid(mask, T)
    sid = np.asarray(seq_id, np.int64)
    if np.any(sid < 0) or np.any(sid >= n_seq):
        raise ValueError("sequence id outside [0, n_seq)")
    if not np.all(np.isfinite(d32[valid])) or np.any(np.abs(d32[valid]) > D_MAX):
        raise ValueError("token log-ratio outside [-128, 128]")
    n_i = np.zeros(n_seq, np.int64)
    d_sum = np.zeros(n_seq)
    for t in range(T):
        if valid[t]:
            n_i[sid[t]] += 1
            d_sum[sid[t]] += float(d32[t])
    S = int(np.sum(n_i > 0))
    lo32, hi32 = np.float32(lo), np.float32(hi)
    s64 = np.zeros(n_seq)
    s32 = np.zeros(n_seq, np.float32)
    cm = np.zeros(n_seq, np.uint8)
    terms = np.zeros(n_seq)
    coef = np.zeros(n_seq)  # g_t of the sequence's valid tokens
    for i in range(n_seq):
        if n_i[i] == 0:
            continue
        s64[i] = np.exp(d_sum[i] / n_i[i])
        s32[i] = np.float32(s64[i])
        A = a_seq[i]
        up = A > 0 and s32[i] >= hi32
        dn = A < 0 and s32[i] <= lo32
        cm[i] = CLIP_HI * up + CLIP_LO * dn
        s = float(s32[i])
        m = min(s, float(hi32)) if A >= 0 else max(s, float(lo32))
        terms[i] = -A * m
        if not (up or dn):
            coef[i] = -A * s / (n_i[i] * S)
    grad = np.zeros(T)
    for t in range(T):
        if valid[t]:
            grad[t] = coef[sid[t]]
    live = n_i > 0
    loss_sum = float(np.sum(terms[live]))
    n_pos = int(np.sum(live & (a_seq > 0)))
    n_neg = int(np.sum(live & (a_seq < 0)))
    c_pos = int(np.sum((cm & CLIP_HI) != 0))
    c_neg = int(np.sum((cm & CLIP_LO) != 0))
    return {
        "loss": loss_sum / S if S else 0.0, "loss_sum": loss_sum, "grad": grad,
        "seq_ratio": s64, "seq_ratio32": s32, "seq_clip": cm, "seq_terms": terms,
        "seq_valid_tokens": n_i, "n_seq_valid": S, "n_valid": int(valid.sum()),
        "n_pos": n_pos, "n_neg": n_neg, "clipped_pos": c_pos, "clipped_neg": c_neg,
        # clip fractions over responses (the unit this variant clips)
        "clip_frac_pos": c_pos / n_pos if n_pos else 0.0,
        "clip_frac_neg": c_neg / n_neg if n_neg else 0.0,
        "clip_frac": (c_pos + c_neg) / S if S else 0.0,
    }
