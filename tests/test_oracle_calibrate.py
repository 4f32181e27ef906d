"""Pins for the oracle's Calibrated Clipping (§4, Eq. 5, Algorithm 1).

* identical FP8 and BF16 ratios return the reference bounds unchanged (both
  modes, GRPO and DAPO reference bounds);
* the calibrated lower bound equalises the number of lower-clipped negative
  tokens (the property §4 states for L = F^-1(alpha_low));
* brute force over every threshold that can matter on tiny inputs (a
  different algorithm from the oracle's interval construction), for L and for
  H, the latter against rho computed in exact rational arithmetic from the
  unrounded Eq. 5 terms;
* GRID mode (Algorithm 1 as printed) by brute force over the grid in exact
  rational arithmetic, on ratios placed exactly on grid points so that the
  strict "<" of Eq. 5 and the tie-breaks decide the answer, and planted slips
  of those rules caught;
* a hand-worked example and SmoothUpdate values with the paper's constants;
* degenerate inputs and the overflow bound of the fixed-point sums.
"""

import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import calibrate as C
from paper_2609_22870_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
F32 = np.float32


def _inputs(T, seed, sigma_fp8=0.05, tie_every=0, frac_zero_adv=0.1):
    r_bf, r_fp, coef = (a.numpy() for a in synth.ratio_inputs(T, seed, sigma_fp8=sigma_fp8,
                                                              tie_every=tie_every))
    rng = np.random.default_rng(seed)
    adv = rng.standard_normal(T).astype(np.float32)
    adv[rng.random(T) < frac_zero_adv] = 0
    mask = (rng.random(T) < 0.9).astype(np.uint8)
    return r_fp, r_bf, adv, mask, coef


@pytest.mark.parametrize("mode", [C.EXACT, C.GRID])
@pytest.mark.parametrize("eps", [(0.2, 0.2), (0.2, 0.28), (0.2, 0.24)])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_identical_ratios_return_reference_bounds(mode, eps, seed):
    r_fp, r_bf, adv, mask, coef = _inputs(4000, seed)
    res = C.calibrate_clip_bounds(r_bf, r_bf, adv, mask, coef, eps[0], eps[1], {"mode": mode})
    c_lo, c_hi = C.reference_bounds(*eps)
    assert res["lo_star"] == c_lo and res["hi_star"] == c_hi
    assert res["k_fp8"] == res["k_bf16"]
    assert res["rho_fp8"] == res["rho_bf16"]


@pytest.mark.parametrize("seed", range(6))
def test_lower_bound_equalises_clipped_counts(seed):
    r_fp, r_bf, adv, mask, coef = _inputs(20000, 100 + seed, sigma_fp8=0.03)
    res = C.calibrate_clip_bounds(r_fp, r_bf, adv, mask, coef, 0.2, 0.2)
    assert 0.5 < res["lo_star"] < 0.9  # unclamped, continuous ratios: no ties
    assert res["k_fp8"] == res["k_bf16"]
    neg = (mask != 0) & (adv < 0)
    assert int(np.sum(neg & (r_fp <= res["lo_star"]))) == res["k_bf16"]


def _brute_lower(r_neg, k, c_lo, lo_min, lo_max):
    """Enumerate every threshold at which #{r <= L} can change, plus c_lo."""
    pts = set()
    for v in list(r_neg) + [c_lo, lo_min, lo_max]:
        v = F32(v)
        pts.update([v, np.nextafter(v, F32(-np.inf)), np.nextafter(v, F32(np.inf))])
    pts = sorted(p for p in pts if lo_min <= p <= lo_max)
    f = {p: abs(int(np.sum(r_neg <= p)) - k) for p in pts}
    fmin = min(f.values())
    best = [p for p in pts if f[p] == fmin]
    return fmin, min(abs(float(p) - float(c_lo)) for p in best), f


@pytest.mark.parametrize("seed", range(40))
def test_lower_bound_brute_force_tiny(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 13))
    r_neg = F32(np.round(rng.uniform(0.4, 1.2, n), int(rng.integers(1, 4))))  # ties likely
    r_bf = F32(np.round(rng.uniform(0.6, 1.0, n), 2))
    adv = -np.ones(n, np.float32)
    res = C.calibrate_clip_bounds(r_neg, r_bf, adv, np.ones(n, np.uint8), None, 0.2, 0.2)
    c_lo = C.reference_bounds(0.2, 0.2)[0]
    k = int(np.sum(r_bf <= c_lo))
    fmin, dist, f = _brute_lower(r_neg, k, c_lo, F32(0.5), F32(0.9))
    L = res["lo_star"]
    assert abs(int(np.sum(r_neg <= L)) - k) == fmin
    assert abs(float(L) - float(c_lo)) == dist


def _rho_exact(r, coef, adv, sel_pos, sel_neg):
    def term(i):
        return Fraction(float(coef[i])) * Fraction(float(r[i])) * Fraction(float(adv[i]))
    num = abs(sum((term(i) for i in sel_pos), Fraction(0)))
    den = abs(sum((term(i) for i in sel_neg), Fraction(0)))
    return num, den


@pytest.mark.parametrize("seed", range(40))
def test_upper_bound_brute_force_tiny(seed):
    rng = np.random.default_rng(1000 + seed)
    n = int(rng.integers(4, 14))
    adv = F32(rng.choice([-1.5, -1.0, -0.5, 0.5, 1.0, 2.0], n))
    adv[0], adv[1] = -1.0, 1.0
    r_bf = F32(rng.uniform(0.7, 1.5, n))
    r_fp = F32(np.round(rng.uniform(0.6, 2.2, n), int(rng.integers(1, 4))))
    coef = F32(rng.uniform(0.1, 1.0, n))
    mask = np.ones(n, np.uint8)
    res = C.calibrate_clip_bounds(r_fp, r_bf, adv, mask, coef, 0.2, 0.2)
    if res["flags"]:
        return
    c_lo, c_hi = C.reference_bounds(0.2, 0.2)
    L, H = res["lo_star"], res["hi_star"]
    pos, neg = np.where(adv > 0)[0], np.where(adv < 0)[0]
    nb, db = _rho_exact(r_bf, coef, adv, [i for i in pos if r_bf[i] < c_hi], [i for i in neg if r_bf[i] > c_lo])
    rho_bf = nb / db
    _, dfp = _rho_exact(r_fp, coef, adv, [], [i for i in neg if r_fp[i] > L])

    def obj(h):
        p, _ = _rho_exact(r_fp, coef, adv, [i for i in pos if r_fp[i] < h], [])
        return abs(p / dfp - rho_bf)

    pts = set()
    for v in list(r_fp[pos]) + [c_hi, 1.2, 2.0]:
        v = F32(v)
        pts.update([v, np.nextafter(v, F32(np.inf))])
    pts = sorted(p for p in pts if F32(1.2) <= p <= F32(2.0))
    objs = {p: obj(p) for p in pts}
    best = min(objs.values())
    got = obj(H)
    # exact up to the fixed-point rounding of the terms (relative 2^-40 or better)
    assert got <= best + abs(rho_bf) * Fraction(1, 2 ** 30)
    if got == best:
        ties = [p for p in pts if objs[p] == best]
        assert abs(float(H) - float(c_hi)) <= min(abs(float(p) - float(c_hi)) for p in ties)


def _golden_rows(name):
    rows, exp = [], {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.split("#")[0].strip()
        if not line:
            continue
        parts = line.split()
        if parts[0].startswith("lo_") or parts[0].startswith("hi_"):
            exp[parts[0]] = parts[1]
        else:
            rows.append([float(x) for x in parts])
    return np.array(rows), exp


def test_hand_worked_example():
    rows, exp = _golden_rows("calib_tiny.txt")
    r_bf, r_fp, adv = (F32(rows[:, i]) for i in range(3))
    mask = np.ones(len(adv), np.uint8)
    ex = C.calibrate_clip_bounds(r_fp, r_bf, adv, mask, None, 0.2, 0.2, {"mode": C.EXACT})
    gr = C.calibrate_clip_bounds(r_fp, r_bf, adv, mask, None, 0.2, 0.2, {"mode": C.GRID})
    assert exp["lo_star_exact"] == "nextbelow(0.74)"
    assert ex["lo_star"] == np.nextafter(F32(0.74), F32(-np.inf))
    assert gr["lo_star"] == F32(float(exp["lo_star_grid"]))
    assert ex["k_bf16"] == 3 and ex["k_fp8"] == 3
    assert ex["flags"] & C.FLAG_NO_POS


def test_smooth_update_golden():
    for line in open(os.path.join(GOLDEN, "smooth_update.txt")):
        line = line.split("#")[0].strip()
        if not line:
            continue
        b, bs, d, e = (float(x) for x in line.split())
        assert C.smooth_update(b, bs, d) == F32(e) or abs(C.smooth_update(b, bs, d) - F32(e)) <= 1.5e-7


def test_smooth_update_applied_to_results():
    r_fp, r_bf, adv, mask, coef = _inputs(5000, 9, sigma_fp8=0.08)
    res = C.calibrate_clip_bounds(r_fp, r_bf, adv, mask, coef, 0.2, 0.2, {"lo_old": 0.6, "hi_old": 1.8})
    assert res["lo_new"] == C.smooth_update(0.6, res["lo_star"], 0.05)
    assert res["hi_new"] == C.smooth_update(1.8, res["hi_star"], 0.1)
    # the step is limited to delta (up to the float32 rounding of b + d)
    assert abs(float(res["lo_new"]) - 0.6) <= 0.05 + 1e-6
    assert abs(float(res["hi_new"]) - 1.8) <= 0.1 + 1e-6


def test_degenerate_inputs():
    r = np.ones(8, np.float32)
    adv = np.ones(8, np.float32)
    res = C.calibrate_clip_bounds(r, r, adv, np.ones(8, np.uint8), None, 0.2, 0.2)
    assert res["flags"] & C.FLAG_NO_NEG and res["lo_star"] == F32(0.8)
    assert res["hi_star"] == F32(1.2)
    res = C.calibrate_clip_bounds(r, r, -adv, np.ones(8, np.uint8), None, 0.2, 0.2)
    assert res["flags"] & C.FLAG_NO_POS and res["hi_star"] == F32(1.2)
    res = C.calibrate_clip_bounds(r, r, adv, np.zeros(8, np.uint8), None, 0.2, 0.2)
    assert res["flags"] & C.FLAG_NO_NEG and res["flags"] & C.FLAG_NO_POS
    # n_valid counts valid tokens of any advantage sign (zero included): here
    # tokens 0, 2, 3 and 5 are valid, with A = +1, -1, 0, 0
    a = np.array([1, 5, -1, 0, 2, 0, 3, 4], np.float32)
    m = np.array([1, 0, 1, 1, 0, 1, 0, 0], np.uint8)
    res = C.calibrate_clip_bounds(r, r, a, m, None, 0.2, 0.2)
    assert (res["n_valid"], res["n_pos"], res["n_neg"]) == (4, 1, 1)
    assert C.calibrate_clip_bounds(r, r, a, None, None, 0.2, 0.2)["n_valid"] == 8


@pytest.mark.parametrize("scale", [1e-30, 1e-5, 1.0, 1e5, 1e30])
def test_fixed_point_sums_never_overflow(scale):
    r_fp, r_bf, adv, mask, coef = _inputs(3000, 5)
    coef = F32(coef / coef.max() * scale)
    res = C.calibrate_clip_bounds(r_fp, r_bf, adv, mask, coef, 0.2, 0.2)
    for key in ("sum_pos_bf16", "sum_neg_bf16", "sum_neg_fp8", "sum_pos_fp8"):
        assert 0 <= res[key] < 2 ** 62
    e = C.update_terms(coef, r_bf, adv)[(mask != 0) & (adv != 0)]
    assert res["shift"] == C.fixed_shift(max(np.abs(e).max(), np.abs(C.update_terms(coef, r_fp, adv)[(mask != 0) & (adv != 0)]).max()),
                                         int(np.sum((mask != 0) & (adv != 0))))
    assert math.ldexp(float(np.abs(e).max()), res["shift"]) * len(e) <= 2.0 ** 62


# ---------------------------------------------------------------- GRID mode
# Algorithm 1 as printed: candidates on the 0.02 grid of I_L and I_H.  The
# brute force below restates the search from the paper directly: every grid
# candidate is scored in exact rational arithmetic (lower: |#{r <= L} - k|;
# upper: |rho_FP8(L*, H) - rho_BF16| with the strict "<" of Eq. 5), the
# minimisers are kept, and the tie goes to the candidate nearest the reference
# bound, then to the smaller one.  Ratios sit exactly on grid points (and one
# float32 step either side), coefficients and advantages are short dyadic
# numbers, so every Eq. 5 term is exact in the oracle's fixed point and a tie
# in the rational objective is a tie there too.  A slip such as "<=" for "<"
# in P(H), or a reversed tie-break, changes the answer on these inputs.

def _grid_points(lo_pct, hi_pct):
    """fl32(k / 100) for the grid's percent values (computed independently of
    the oracle's fl32(lo + i * step))."""
    return [F32(p / 100) for p in range(lo_pct, hi_pct + 1, 2)]


def _on_grid_ratios(rng, n, pts):
    out = []
    for _ in range(n):
        v = pts[int(rng.integers(0, len(pts)))]
        how = int(rng.integers(0, 4))
        if how == 1:
            v = np.nextafter(v, F32(np.inf))
        elif how == 2:
            v = np.nextafter(v, F32(-np.inf))
        out.append(v)
    return F32(out)


def _brute_grid(r_fp, r_bf, adv, coef, c_lo, c_hi, lo_pts, hi_pts):
    neg = [i for i in range(len(adv)) if adv[i] < 0]
    pos = [i for i in range(len(adv)) if adv[i] > 0]
    k = sum(1 for i in neg if r_bf[i] <= c_lo)

    def pick(cands, key, ref):
        best = min(key(c) for c in cands)
        ties = [c for c in cands if key(c) == best]
        return min(ties, key=lambda c: (abs(Fraction(float(c)) - Fraction(float(ref))), float(c)))

    L = pick(lo_pts, lambda c: abs(sum(1 for i in neg if r_fp[i] <= c) - k), c_lo)

    def e(i, r):
        return Fraction(float(coef[i])) * Fraction(float(r[i])) * Fraction(float(adv[i]))

    n_bf = abs(sum((e(i, r_bf) for i in pos if r_bf[i] < c_hi), Fraction(0)))
    d_bf = abs(sum((e(i, r_bf) for i in neg if r_bf[i] > c_lo), Fraction(0)))
    d_fp = abs(sum((e(i, r_fp) for i in neg if r_fp[i] > L), Fraction(0)))
    if not pos or d_bf == 0 or d_fp == 0:
        return L, None
    rho_bf = n_bf / d_bf

    def obj(c):
        p = sum((e(i, r_fp) for i in pos if r_fp[i] < c), Fraction(0))
        return abs(p / d_fp - rho_bf)

    return L, pick(hi_pts, obj, c_hi)


def _grid_case(seed):
    rng = np.random.default_rng(7000 + seed)
    n = int(rng.integers(5, 16))
    lo_pts, hi_pts = _grid_points(50, 90), _grid_points(120, 200)
    adv = F32(rng.choice([-2.0, -1.0, -0.5, 0.5, 1.0, 1.5], n))
    adv[0], adv[1] = -1.0, 1.0
    coef = F32(rng.choice([0.25, 0.5, 1.0, 2.0], n))
    r_fp = _on_grid_ratios(rng, n, lo_pts + hi_pts)
    r_bf = _on_grid_ratios(rng, n, lo_pts + hi_pts)
    eps_hi = [0.2, 0.28, 0.24][seed % 3]
    return r_fp, r_bf, adv, coef, eps_hi, lo_pts, hi_pts


@pytest.mark.parametrize("seed", range(60))
def test_grid_bounds_brute_force_on_grid_ratios(seed):
    r_fp, r_bf, adv, coef, eps_hi, lo_pts, hi_pts = _grid_case(seed)
    res = C.calibrate_clip_bounds(r_fp, r_bf, adv, np.ones(len(adv), np.uint8), coef, 0.2, eps_hi,
                                  {"mode": C.GRID})
    c_lo, c_hi = C.reference_bounds(0.2, eps_hi)
    L, H = _brute_grid(r_fp, r_bf, adv, coef, c_lo, c_hi, lo_pts, hi_pts)
    assert res["lo_star"] == L
    if H is None:
        assert res["flags"] & (C.FLAG_NO_POS | C.FLAG_ZERO_D_BF16 | C.FLAG_ZERO_D_FP8)
    else:
        assert res["flags"] == 0
        assert res["hi_star"] == H


def test_grid_candidates_match_percent_values():
    """The oracle's fl32(lo + i * step) grid is the float32 of k/100."""
    assert C.grid(0.5, 0.9, 0.02) == _grid_points(50, 90)
    assert C.grid(1.2, 2.0, 0.02) == _grid_points(120, 200)


def test_grid_brute_force_catches_planted_slips(monkeypatch):
    """Plant the slips the pin must catch into the oracle (on the CPU) and
    require that the brute force disagrees on at least one case each."""
    def le_instead_of_lt(r_pos, q_pos, d_bf, x, c_hi, cands):
        r_pos = np.asarray(r_pos, np.float32)
        q_pos = np.asarray(q_pos, np.int64)
        best = None
        for c in cands:
            p = C._isum(q_pos[r_pos <= c])
            key = (abs(p * d_bf - x), abs(float(c) - float(c_hi)), float(c))
            if best is None or key < best[0]:
                best = (key, c)
        return np.float32(best[1])

    def far_tie_break(r_pos, q_pos, d_bf, x, c_hi, cands):
        r_pos = np.asarray(r_pos, np.float32)
        q_pos = np.asarray(q_pos, np.int64)
        best = None
        for c in cands:
            p = C._isum(q_pos[r_pos < c])
            key = (abs(p * d_bf - x), -abs(float(c) - float(c_hi)), float(c))
            if best is None or key < best[0]:
                best = (key, c)
        return np.float32(best[1])

    for slip in (le_instead_of_lt, far_tie_break):
        monkeypatch.setattr(C, "upper_bound_grid", slip)
        caught = 0
        for seed in range(60):
            r_fp, r_bf, adv, coef, eps_hi, lo_pts, hi_pts = _grid_case(seed)
            res = C.calibrate_clip_bounds(r_fp, r_bf, adv, np.ones(len(adv), np.uint8), coef, 0.2, eps_hi,
                                          {"mode": C.GRID})
            c_lo, c_hi = C.reference_bounds(0.2, eps_hi)
            _, H = _brute_grid(r_fp, r_bf, adv, coef, c_lo, c_hi, lo_pts, hi_pts)
            caught += H is not None and res["hi_star"] != H
        assert caught > 0, slip.__name__
        monkeypatch.undo()


def test_grid_brute_force_catches_planted_lower_slips(monkeypatch):
    """The same for the lower bound: "<" for the CDF's "<=", and the tie going
    to the larger candidate instead of the one nearer c_low."""
    def lt_instead_of_le(r_neg, k, c_lo, cands):
        r_neg = np.asarray(r_neg, np.float32)
        best = None
        for c in cands:
            key = (abs(int(np.sum(r_neg < c)) - k), abs(float(c) - float(c_lo)), float(c))
            if best is None or key < best[0]:
                best = (key, c)
        return np.float32(best[1])

    def larger_first(r_neg, k, c_lo, cands):
        r_neg = np.asarray(r_neg, np.float32)
        best = None
        for c in cands:
            key = (abs(int(np.sum(r_neg <= c)) - k), -float(c))
            if best is None or key < best[0]:
                best = (key, c)
        return np.float32(best[1])

    for slip in (lt_instead_of_le, larger_first):
        monkeypatch.setattr(C, "lower_bound_grid", slip)
        caught = 0
        for seed in range(60):
            r_fp, r_bf, adv, coef, eps_hi, lo_pts, hi_pts = _grid_case(seed)
            res = C.calibrate_clip_bounds(r_fp, r_bf, adv, np.ones(len(adv), np.uint8), coef, 0.2, eps_hi,
                                          {"mode": C.GRID})
            c_lo, c_hi = C.reference_bounds(0.2, eps_hi)
            L, _ = _brute_grid(r_fp, r_bf, adv, coef, c_lo, c_hi, lo_pts, hi_pts)
            caught += res["lo_star"] != L
        assert caught > 0, slip.__name__
        monkeypatch.undo()
