"""Over-clipping, PPO clip fractions and NMAE diagnostics (§3); TIS weights (§2.3).

Test infrastructure only (see ``oracle/__init__.py``).

§3 ("The Cause") diagnoses full-pipeline FP8 instability against BF16 shadow
passes:

* the normalised mean absolute error of the FP8-induced probabilities and of
  the importance ratios relative to their BF16 references,
      NMAE(x, x_ref) = sum |x - x_ref| / sum |x_ref|      (valid tokens)
  (the paper reports the ratio NMAE 1.7x to 2.9x the probability NMAE);
* over-clipping: a token is lower-bound over-clipped if A < 0,
  r_BF16 > 1 - eps and r_FP8 <= 1 - eps, upper-bound over-clipped if A > 0,
  r_BF16 < 1 + eps and r_FP8 >= 1 + eps;
* the PPO clip fractions of the FP8 and of the BF16 ratios at the same bounds
  (clipped at equality, §2.1).

The truncated importance-sampling weight of J_TIS (§2.3) is
      w_t = min(pi_old(y_t|h_t) / pi_sampler(y_t|h_t), C),   C = 2 typically.

Readings: the bounds are the float32 values fl32(1 - eps_low) and
fl32(1 + eps_high), as in calibration; a probability is exp(logp) of the
sampled token; a token counts iff mask = 1 and A = 0 tokens belong to neither
sign; pi_old / pi_sampler = exp(logp_old - logp_sampler).  Everything is
evaluated in float64 from the float32 inputs, counts exactly.
"""

import numpy as np


def tis_weights(logp_old, logp_sampler, C=2.0):
    """w_t = min(exp(logp_old - logp_sampler), C) in float64 (§2.3, J_TIS)."""
    lo = np.asarray(logp_old, np.float32).astype(np.float64)
    ls = np.asarray(logp_sampler, np.float32).astype(np.float64)
    return np.minimum(np.exp(lo - ls), float(C))


def nmae(x, ref):
    """sum |x - ref| / sum |ref| (NaN when the reference sums to zero)."""
    x = np.asarray(x, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.sum(np.abs(ref))
    return np.sum(np.abs(x - ref)) / den if den > 0 else np.nan


def clip_diagnostics(logp_fp8, logp_bf16, r_fp8, r_bf16, adv, mask, eps_low, eps_high):
    """Counts and NMAEs of §3 over the valid tokens.  logp_* may be None (no
    probability NMAE)."""
    r8 = np.asarray(r_fp8, np.float32)
    rb = np.asarray(r_bf16, np.float32)
    A = np.asarray(adv, np.float32)
    valid = np.ones(r8.shape, bool) if mask is None else np.asarray(mask) != 0
    c_lo = np.float32(np.float32(1.0) - np.float32(eps_low))
    c_hi = np.float32(np.float32(1.0) + np.float32(eps_high))
    neg = valid & (A < 0)
    pos = valid & (A > 0)
    out = {
        "c_lo": c_lo, "c_hi": c_hi,
        "n_valid": int(valid.sum()), "n_pos": int(pos.sum()), "n_neg": int(neg.sum()),
        "clipped_lo_fp8": int((neg & (r8 <= c_lo)).sum()),
        "clipped_hi_fp8": int((pos & (r8 >= c_hi)).sum()),
        "clipped_lo_bf16": int((neg & (rb <= c_lo)).sum()),
        "clipped_hi_bf16": int((pos & (rb >= c_hi)).sum()),
        "over_clipped_lo": int((neg & (rb > c_lo) & (r8 <= c_lo)).sum()),
        "over_clipped_hi": int((pos & (rb < c_hi) & (r8 >= c_hi)).sum()),
    }
    r8v, rbv = r8[valid].astype(np.float64), rb[valid].astype(np.float64)
    out["abs_err_ratio"] = float(np.sum(np.abs(r8v - rbv)))
    out["sum_ratio_bf16"] = float(np.sum(np.abs(rbv)))
    out["nmae_ratio"] = nmae(r8v, rbv)
    if logp_fp8 is not None and logp_bf16 is not None:
        p8 = np.exp(np.asarray(logp_fp8, np.float32)[valid].astype(np.float64))
        pb = np.exp(np.asarray(logp_bf16, np.float32)[valid].astype(np.float64))
        out["abs_err_prob"] = float(np.sum(np.abs(p8 - pb)))
        out["sum_prob_bf16"] = float(np.sum(pb))
        out["nmae_prob"] = nmae(p8, pb)
    else:
        out["abs_err_prob"] = out["sum_prob_bf16"] = 0.0
        out["nmae_prob"] = np.nan
    return out
