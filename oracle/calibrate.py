"""Calibrated Clipping (§4, Eq. 5, Algorithm 1) -- oracle side.

Test infrastructure only (see ``oracle/__init__.py``).

What the paper fixes
--------------------
* Lower-bound alignment (§4, stage 1): over tokens with A_t < 0,
  alpha_low = F_BF16,-(1 - eps) and L = F_FP8,-^{-1}(alpha_low), which makes the
  number of lower-clipped tokens equal under both precisions.
* Upper-bound rebalancing (§4, stage 2, Eq. 5):
      rho = |sum_{A>0} w pi_s r A 1{r < c_high}| / |sum_{A<0} w pi_s r A 1{r > c_low}|
  rho_BF16 from the BF16 ratios at the reference bounds; H solves
  rho_FP8(L, H) = rho_BF16.
* Algorithm 1: grid search of L* in I_L = [0.5, 0.9] and H* in I_H = [1.2, 2.0]
  with step 0.02, minimising |F_FP8,-(L*) - alpha_low| and
  |rho_FP8(L*, H*) - rho_BF16|; then SmoothUpdate(b, b*, d) =
  b + clip((b* - b)/2, -d, d) with d_L = 0.05, d_H = 0.1; initial bounds
  [0.6, 1.8].
* Clip semantics at equality (§2.1): A > 0 is clipped when r >= 1 + eps, A < 0
  when r <= 1 - eps, hence F(x) counts r <= x, and the "unclipped" indicators of
  Eq. 5 are strict (r < c_high, r > c_low).

Readings taken where the paper is silent or set-valued
------------------------------------------------------
* Valid tokens: mask = 1.  A = 0 tokens belong to neither sign set.
* c_low = fl32(1 - eps_low), c_high = fl32(1 + eps_high).
* k = #{Neg : r_bf16 <= c_low}; alpha_low = k / |Neg|.
* EXACT mode (default): F_FP8,- is a step function, so its inverse at alpha_low
  is an interval of thresholds.  Over all float32 thresholds L in I_L,
  |#{Neg: r_fp8 <= L} - k| is minimised on one interval; L* is the point of
  that interval closest to c_low.  (With identical FP8 and BF16 ratios this
  returns c_low unchanged.)  This is Algorithm 1's search over I_L with the
  grid refined to every float32.
* GRID mode (Algorithm 1 as printed): candidates fl32(I_lo + i * step) computed
  in float64; ties go to the candidate closer to the reference bound, then to the
  smaller one.
* Eq. 5 terms: e_t = (coef_t * r_t) * A_t in float64 with coef_t = w_t^TIS *
  pi_sampler(y_t | h_t) (the caller supplies the product; nullable => 1).  Eq. 5
  uses pi_sampler where the decomposition of §2.1 uses pi_old; we follow Eq. 5.
* Sums are exact: each e_t becomes the integer q_t = RNE(e_t * 2**s), with one
  shift s per call chosen from the data so that no sum can overflow 62 bits:
  s = 62 - E - B, where max|e| < 2**E and 2**B >= number of signed tokens.  The
  objective |P(H) * D_bf - N_bf * D_fp8| is then compared exactly (it is
  |rho_FP8 - rho_BF16| scaled by the positive constant D_bf * D_fp8).
* EXACT mode for H: P(H) = sum_{Pos, r_fp8 < H} q is a step function of H; over
  all float32 H in I_H the objective is minimised on one interval; H* is its
  point closest to c_high.
* rho_FP8 uses L* (the searched bound, before smoothing), as Algorithm 1 writes
  rho_FP8(L*, H*).
* Degenerate inputs: |Neg| = 0 gives L* = clamp(c_low, I_L); |Pos| = 0,
  D_bf = 0 or D_fp8 = 0 gives H* = clamp(c_high, I_H); each sets a flag.
* SmoothUpdate runs in float32 in the order d = (b* - b) * 0.5; d = min(max(d,
  -delta), delta); b + d.  A NaN previous bound means "no previous bound" and
  returns b* unchanged.
"""

import math

import numpy as np

EXACT, GRID = 0, 1

FLAG_NO_NEG = 1
FLAG_NO_POS = 2
FLAG_ZERO_D_BF16 = 4
FLAG_ZERO_D_FP8 = 8

DEFAULTS = {
    "mode": EXACT,
    "lo_min": 0.5, "lo_max": 0.9,     # I_L
    "hi_min": 1.2, "hi_max": 2.0,     # I_H
    "step": 0.02,                     # Delta
    "delta_lo": 0.05, "delta_hi": 0.1,
    "lo_old": float("nan"), "hi_old": float("nan"),
}

F32_INF = np.float32(np.inf)


def reference_bounds(eps_low, eps_high):
    """(c_low, c_high) = (fl32(1 - eps_low), fl32(1 + eps_high))."""
    one = np.float32(1.0)
    return one - np.float32(eps_low), one + np.float32(eps_high)


def update_terms(coef, r, adv):
    """e_t = (coef_t * r_t) * A_t in float64 (the summand of Eq. 5)."""
    return (np.asarray(coef, np.float64) * np.asarray(r, np.float64)) * np.asarray(adv, np.float64)


def fixed_shift(emax, n_terms):
    """Shift s = 62 - E - B so every sum of q_t = RNE(e_t 2^s) fits in 62 bits.

    ``emax`` is max |e_t| over the signed tokens of both precisions, ``n_terms``
    the number of signed tokens (|Neg| + |Pos|); emax < 2**E, 2**B >= n_terms.
    """
    emax = float(emax)
    if n_terms == 0 or emax == 0.0:
        return 0
    E = math.frexp(emax)[1]          # emax = f * 2**E, f in [0.5, 1)
    B = (int(n_terms) - 1).bit_length()
    return 62 - E - B


def to_fixed(e, s):
    """q_t = RNE(e_t * 2**s) as exact Python-compatible int64."""
    return np.rint(np.ldexp(np.asarray(e, np.float64), s)).astype(np.int64)


def _isum(q):
    return int(sum(int(v) for v in q))


def _pick(cand, target, lo_min, lo_max):
    """Among candidate pieces (f, a, b) -- closed float32 intervals [a, b] on
    which the objective equals f -- keep the parts inside [lo_min, lo_max],
    take those with the least f (they form one interval, the objective being
    unimodal), and return the point of that interval nearest ``target``."""
    kept = []
    for f, a, b in cand:
        a2, b2 = max(a, lo_min), min(b, lo_max)
        if a2 <= b2:
            kept.append((f, a2, b2))
    fmin = min(f for f, _, _ in kept)
    sel = [(a, b) for f, a, b in kept if f == fmin]
    lo, hi = min(a for a, _ in sel), max(b for _, b in sel)
    for (a0, b0), (a1, b1) in zip(sel, sel[1:]):
        assert a1 <= np.nextafter(b0, F32_INF), "minimisers not contiguous"
    return np.float32(min(max(target, lo), hi))


def lower_bound_exact(r_neg, k, c_lo, lo_min, lo_max):
    """Point nearest c_low of the L in I_L minimising |#{Neg: r_fp8 <= L} - k|.

    #{r <= L} is constant on [u_i, u_{i+1}) between consecutive distinct ratio
    values u_i (and equals 0 below u_1); each such piece is one candidate.
    """
    v = np.sort(np.asarray(r_neg, np.float32))
    uniq = np.unique(v)
    cle = np.searchsorted(v, uniq, side="right")
    ninf = -F32_INF
    cand = [(k, ninf, np.nextafter(uniq[0], ninf) if uniq.size else F32_INF)]
    for i in range(uniq.size):
        hi = np.nextafter(uniq[i + 1], ninf) if i + 1 < uniq.size else F32_INF
        cand.append((abs(int(cle[i]) - k), uniq[i], hi))
    return _pick(cand, c_lo, np.float32(lo_min), np.float32(lo_max))


def upper_bound_exact(r_pos, q_pos, d_bf, x, c_hi, hi_min, hi_max):
    """Point nearest c_high of the H in I_H minimising |P(H) d_bf - x|.

    P(H) = sum_{Pos, r_fp8 < H} q is constant on (u_i, u_{i+1}] between
    consecutive distinct ratio values (and equals 0 for H <= u_1).
    """
    r_pos = np.asarray(r_pos, np.float32)
    order = np.argsort(r_pos, kind="stable")
    v = r_pos[order]
    w = np.asarray(q_pos, np.int64)[order]
    uniq = np.unique(v)
    cand = [(abs(x), -F32_INF, uniq[0] if uniq.size else F32_INF)]
    p = 0
    j = 0
    for i in range(uniq.size):
        while j < v.size and v[j] == uniq[i]:
            p += int(w[j])
            j += 1
        hi = uniq[i + 1] if i + 1 < uniq.size else F32_INF
        cand.append((abs(p * d_bf - x), np.nextafter(uniq[i], F32_INF), hi))
    return _pick(cand, c_hi, np.float32(hi_min), np.float32(hi_max))


def grid(lo, hi, step):
    """Algorithm 1 search grid: fl32(lo + i * step), i = 0 .. round((hi-lo)/step)."""
    n = int(round((hi - lo) / step)) + 1
    return [np.float32(lo + i * step) for i in range(n)]


def lower_bound_grid(r_neg, k, c_lo, cands):
    r_neg = np.asarray(r_neg, np.float32)
    best = None
    for c in cands:
        key = (abs(int(np.sum(r_neg <= c)) - k), abs(float(c) - float(c_lo)), float(c))
        if best is None or key < best[0]:
            best = (key, c)
    return np.float32(best[1])


def upper_bound_grid(r_pos, q_pos, d_bf, x, c_hi, cands):
    r_pos = np.asarray(r_pos, np.float32)
    q_pos = np.asarray(q_pos, np.int64)
    best = None
    for c in cands:
        p = _isum(q_pos[r_pos < c])
        key = (abs(p * d_bf - x), abs(float(c) - float(c_hi)), float(c))
        if best is None or key < best[0]:
            best = (key, c)
    return np.float32(best[1])


def smooth_update(b_old, b_star, delta):
    """SmoothUpdate(b, b*, delta) = b + clip((b* - b)/2, -delta, delta), float32."""
    b_old = np.float32(b_old)
    b_star = np.float32(b_star)
    if np.isnan(b_old):
        return b_star
    d = (b_star - b_old) * np.float32(0.5)
    dl = np.float32(delta)
    d = min(max(d, -dl), dl)
    return np.float32(b_old + d)


def calibrate_clip_bounds(r_fp8, r_bf16, adv, mask, coef, eps_low, eps_high, opts=None):
    """Algorithm 1 with the readings above.  Returns a dict of results."""
    o = dict(DEFAULTS)
    if opts:
        o.update(opts)
    r_fp8 = np.asarray(r_fp8, np.float32)
    r_bf16 = np.asarray(r_bf16, np.float32)
    adv = np.asarray(adv, np.float32)
    mask = np.ones(r_fp8.size, bool) if mask is None else np.asarray(mask) != 0
    coef = np.ones_like(r_fp8) if coef is None else np.asarray(coef, np.float32)
    for a in (r_fp8, r_bf16, adv, coef):
        if not np.all(np.isfinite(a)):
            raise ValueError("calibrate: non-finite input")
    if np.any(coef < 0) or np.any(r_fp8 < 0) or np.any(r_bf16 < 0):
        raise ValueError("calibrate: ratios and coef must be >= 0")

    c_lo, c_hi = reference_bounds(eps_low, eps_high)
    neg = mask & (adv < 0)
    pos = mask & (adv > 0)
    n_neg, n_pos = int(neg.sum()), int(pos.sum())
    k = int(np.sum(neg & (r_bf16 <= c_lo)))
    flags = 0

    e_bf = update_terms(coef, r_bf16, adv)
    e_fp = update_terms(coef, r_fp8, adv)
    signed = neg | pos
    emax = max(np.max(np.abs(e_bf[signed]), initial=0.0), np.max(np.abs(e_fp[signed]), initial=0.0))
    s = fixed_shift(emax, n_neg + n_pos)
    q_bf = to_fixed(e_bf, s)
    q_fp = to_fixed(e_fp, s)
    n_bf = _isum(q_bf[pos & (r_bf16 < c_hi)])
    d_bf = abs(_isum(q_bf[neg & (r_bf16 > c_lo)]))

    lo_min, lo_max = np.float32(o["lo_min"]), np.float32(o["lo_max"])
    hi_min, hi_max = np.float32(o["hi_min"]), np.float32(o["hi_max"])

    # Stage 1: lower-bound alignment
    if n_neg == 0:
        flags |= FLAG_NO_NEG
        lo_star = np.float32(min(max(c_lo, lo_min), lo_max))
    elif o["mode"] == GRID:
        lo_star = lower_bound_grid(r_fp8[neg], k, c_lo, grid(o["lo_min"], o["lo_max"], o["step"]))
    else:
        lo_star = lower_bound_exact(r_fp8[neg], k, c_lo, lo_min, lo_max)

    # Stage 2: upper-bound rebalancing
    d_fp = abs(_isum(q_fp[neg & (r_fp8 > lo_star)]))
    x = n_bf * d_fp
    if n_pos == 0:
        flags |= FLAG_NO_POS
    if d_bf == 0:
        flags |= FLAG_ZERO_D_BF16
    if d_fp == 0:
        flags |= FLAG_ZERO_D_FP8
    if flags & (FLAG_NO_POS | FLAG_ZERO_D_BF16 | FLAG_ZERO_D_FP8):
        hi_star = np.float32(min(max(c_hi, hi_min), hi_max))
    elif o["mode"] == GRID:
        hi_star = upper_bound_grid(r_fp8[pos], q_fp[pos], d_bf, x, c_hi,
                                   grid(o["hi_min"], o["hi_max"], o["step"]))
    else:
        hi_star = upper_bound_exact(r_fp8[pos], q_fp[pos], d_bf, x, c_hi, hi_min, hi_max)

    p_fp = _isum(q_fp[pos & (r_fp8 < hi_star)])
    return {
        "lo_star": np.float32(lo_star),
        "hi_star": np.float32(hi_star),
        "lo_new": smooth_update(o["lo_old"], lo_star, o["delta_lo"]),
        "hi_new": smooth_update(o["hi_old"], hi_star, o["delta_hi"]),
        "c_lo": c_lo, "c_hi": c_hi,
        "n_neg": n_neg, "n_pos": n_pos, "k_bf16": k,
        "n_valid": int(mask.sum()),  # every valid token, any advantage (the surrogate's mean)
        "k_fp8": int(np.sum(neg & (r_fp8 <= lo_star))),
        "shift": s,
        "sum_pos_bf16": n_bf, "sum_neg_bf16": d_bf,
        "sum_neg_fp8": d_fp, "sum_pos_fp8": p_fp,
        "rho_bf16": (n_bf / d_bf) if d_bf else float("nan"),
        "rho_fp8": (p_fp / d_fp) if d_fp else float("nan"),
        "flags": flags,
    }
