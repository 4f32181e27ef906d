"""GPU parity: Calibrated Clipping (a5) bit-exact against the oracle.

Both sides select on the same seeded synthetic ratios.  L*, H*, the smoothed
bounds, the counts, the fixed-point shift and every exact sum must match to
the bit; rho is compared to float64 rounding.
"""

import numpy as np
import pytest
import torch

from oracle import calibrate as OC
from paper_2609_22870_gb300 import synth

pytestmark = pytest.mark.gpu


def _inputs(T, seed, sigma_fp8=0.05, tie_every=0, zero_adv=0.1, mask_p=0.9, coef_scale=None):
    r_bf, r_fp, coef = synth.ratio_inputs(T, seed, sigma_fp8=sigma_fp8, tie_every=tie_every)
    g = torch.Generator().manual_seed(seed + 99)
    adv = torch.randn(T, generator=g)
    adv[torch.rand(T, generator=g) < zero_adv] = 0
    mask = (torch.rand(T, generator=g) < mask_p).to(torch.uint8)
    if coef_scale is not None:
        coef = coef / coef.max() * coef_scale
    return r_fp.float(), r_bf.float(), adv.float(), mask, coef.float()


def _run(api, r_fp, r_bf, adv, mask, coef, eps_low, eps_high, **opts):
    d = [None if t is None else t.cuda() for t in (r_fp, r_bf, adv, mask, coef)]
    buf = api.calibrate_clip_bounds(*d, eps_low, eps_high, api.calib_opts(**opts) if opts else None)
    api.check()
    return api.read_calib_result(buf)


def _ref(r_fp, r_bf, adv, mask, coef, eps_low, eps_high, **opts):
    n = lambda t: None if t is None else t.numpy()  # noqa: E731
    return OC.calibrate_clip_bounds(n(r_fp), n(r_bf), n(adv), n(mask), n(coef), eps_low, eps_high, opts)


def _compare(got, ref):
    for k in ("lo_star", "hi_star", "lo_new", "hi_new", "c_lo", "c_hi"):
        assert np.float32(got[k]) == ref[k] or (np.isnan(got[k]) and np.isnan(ref[k])), (k, got[k], ref[k])
    for k in ("n_neg", "n_pos", "n_valid", "k_bf16", "k_fp8", "flags", "shift", "sum_pos_bf16",
              "sum_neg_bf16", "sum_neg_fp8", "sum_pos_fp8"):
        assert got[k] == ref[k], (k, got[k], ref[k])
    for k in ("rho_bf16", "rho_fp8"):
        if np.isnan(ref[k]):
            assert np.isnan(got[k])
        else:
            assert abs(got[k] - ref[k]) <= 1e-12 * max(1.0, abs(ref[k])), (k, got[k], ref[k])


MODES = [OC.EXACT, OC.GRID]


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("T", [1, 2, 17, 1000, 40000, 65537, 200000, 262145])
@pytest.mark.parametrize("eps", [(0.2, 0.2), (0.2, 0.28)])
def test_calibrate_parity(cuda_lib, mode, T, eps):
    args = _inputs(T, T + int(eps[1] * 100))
    _compare(_run(cuda_lib, *args, *eps, mode=mode), _ref(*args, *eps, mode=mode))


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("seed", range(6))
def test_calibrate_wide_noise_hits_interval_ends(cuda_lib, mode, seed):
    """Large FP8 noise pushes the unconstrained optimum outside I_L / I_H."""
    args = _inputs(5000, 300 + seed, sigma_fp8=[0.02, 0.3, 0.6, 1.0, 2.0, 0.1][seed])
    _compare(_run(cuda_lib, *args, 0.2, 0.2, mode=mode), _ref(*args, 0.2, 0.2, mode=mode))


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("tie_every", [2, 7, 1000])
def test_calibrate_ties(cuda_lib, mode, tie_every):
    args = _inputs(6000, 41 + tie_every, tie_every=tie_every)
    _compare(_run(cuda_lib, *args, 0.2, 0.2, mode=mode), _ref(*args, 0.2, 0.2, mode=mode))


@pytest.mark.parametrize("mode", MODES)
def test_calibrate_identity_returns_reference_bounds(cuda_lib, mode):
    r_fp, r_bf, adv, mask, coef = _inputs(20000, 5)
    got = _run(cuda_lib, r_bf, r_bf, adv, mask, coef, 0.2, 0.28, mode=mode)
    c_lo, c_hi = OC.reference_bounds(0.2, 0.28)
    assert np.float32(got["lo_star"]) == c_lo and np.float32(got["hi_star"]) == c_hi


@pytest.mark.parametrize("scale", [1e-30, 1e-6, 1.0, 1e6, 1e30])
def test_calibrate_coef_scales(cuda_lib, scale):
    args = _inputs(3000, 8, coef_scale=scale)
    _compare(_run(cuda_lib, *args, 0.2, 0.2), _ref(*args, 0.2, 0.2))


@pytest.mark.parametrize("mode", MODES)
def test_calibrate_smoothing_and_nullable_inputs(cuda_lib, mode):
    r_fp, r_bf, adv, mask, coef = _inputs(4000, 12, sigma_fp8=0.1)
    kw = dict(mode=mode, lo_old=0.6, hi_old=1.8)
    _compare(_run(cuda_lib, r_fp, r_bf, adv, None, None, 0.2, 0.2, **kw),
             _ref(r_fp, r_bf, adv, None, None, 0.2, 0.2, **kw))


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("case", ["no_neg", "no_pos", "all_masked", "empty", "zero_coef"])
def test_calibrate_degenerate(cuda_lib, mode, case):
    r_fp, r_bf, adv, mask, coef = _inputs(500, 13)
    if case == "no_neg":
        adv = adv.abs()
    elif case == "no_pos":
        adv = -adv.abs()
    elif case == "all_masked":
        mask = torch.zeros_like(mask)
    elif case == "zero_coef":
        coef = torch.zeros_like(coef)
    elif case == "empty":
        r_fp, r_bf, adv, mask, coef = (t[:0] for t in (r_fp, r_bf, adv, mask, coef))
    _compare(_run(cuda_lib, r_fp, r_bf, adv, mask, coef, 0.2, 0.2, mode=mode),
             _ref(r_fp, r_bf, adv, mask, coef, 0.2, 0.2, mode=mode))


def test_calibrate_grid_custom_interval(cuda_lib):
    args = _inputs(8000, 14, sigma_fp8=0.08)
    kw = dict(mode=OC.GRID, lo_min=0.6, lo_max=0.95, hi_min=1.1, hi_max=3.0, step=0.005)
    _compare(_run(cuda_lib, *args, 0.2, 0.2, **kw), _ref(*args, 0.2, 0.2, **kw))


@pytest.mark.parametrize("name", ["grpo_8b", "dapo_32b", "long_8b"])
def test_calibrate_full_size(cuda_lib, name):
    """Token counts and group/mask layouts of the full workloads."""
    w = synth.WORKLOADS[name]
    adv, mask = synth.rollout(w)
    r_bf, r_fp, coef = synth.ratio_inputs(w.T, w.seed, sigma_fp8=0.04)
    for mode in MODES:
        _compare(_run(cuda_lib, r_fp, r_bf, adv, mask, coef, w.eps_low, w.eps_high, mode=mode),
                 _ref(r_fp, r_bf, adv, mask, coef, w.eps_low, w.eps_high, mode=mode))


@pytest.mark.parametrize("mode", MODES)
def test_calibrate_unaligned_inputs(cuda_lib, mode):
    """Inputs that start 4 bytes (1 byte for the mask) past an allocation
    boundary take the scalar-load passes; same result as the oracle."""
    T = 3001
    args = _inputs(T + 1, 77)
    d = [None if t is None else t.cuda()[1:] for t in args]
    buf = cuda_lib.calibrate_clip_bounds(*d, 0.2, 0.28, cuda_lib.calib_opts(mode=mode))
    cuda_lib.check()
    host = [None if t is None else t[1:] for t in args]
    _compare(cuda_lib.read_calib_result(buf), _ref(*host, 0.2, 0.28, mode=mode))


def _interval_case(case, T, seed):
    """Inputs that put the selection on a given side of the search intervals
    I_L = [0.5, 0.9], I_H = [1.2, 2.0]: Algorithm 1 minimises over the pieces
    inside the interval, so a crossing below or above it must come back as the
    piece at that end, and ratios lying exactly on an end must count on the
    right side of it (r <= L for the lower CDF, r < H for P(H))."""
    r_fp, r_bf, adv, mask, coef = _inputs(T, seed)
    g = torch.Generator().manual_seed(seed + 7)
    neg, pos = adv < 0, adv > 0
    if case == "lower_crossing_above_interval":  # C(lo_max) < k: many A<0 with r_bf <= c_lo, none in I_L
        r_bf[neg] = 0.7
        r_fp[neg] = 0.95 + 0.01 * torch.rand(int(neg.sum()), generator=g)
    elif case == "lower_crossing_below_interval":  # k <= C(lo_min^-): most A<0 ratios under lo_min
        r_fp[neg] = 0.3 + 0.1 * torch.rand(int(neg.sum()), generator=g)
    elif case == "upper_target_below_interval":  # P(hi_min) D_bf >= N_bf D_fp8
        r_bf[pos] = 1.1
        r_fp[pos] = 1.15
    elif case == "upper_target_above_interval":  # every A>0 ratio at or above hi_max
        r_fp[pos] = 2.0 + torch.rand(int(pos.sum()), generator=g)
    elif case == "ratios_on_interval_ends":
        ends = torch.tensor([0.5, 0.9, 1.2, 2.0], dtype=torch.float32)
        pick = torch.randint(0, 4, (T,), generator=g)
        on = torch.rand(T, generator=g) < 0.3
        r_fp[on] = ends[pick[on]]
        r_bf[on & (torch.rand(T, generator=g) < 0.5)] = 0.8
    return r_fp, r_bf, adv, mask, coef


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("T", [5000, 300000])
@pytest.mark.parametrize("case", ["lower_crossing_above_interval", "lower_crossing_below_interval",
                                  "upper_target_below_interval", "upper_target_above_interval",
                                  "ratios_on_interval_ends"])
def test_calibrate_crossings_outside_the_interval(cuda_lib, mode, T, case):
    """Both launch paths (one cooperative launch up to 2^18 tokens, stage
    launches above), every side a crossing can fall on, and ratios on the
    interval ends; bit-exact against the oracle."""
    args = _interval_case(case, T, 400 + T % 97)
    _compare(_run(cuda_lib, *args, 0.2, 0.2, mode=mode), _ref(*args, 0.2, 0.2, mode=mode))


@pytest.mark.parametrize("T", [5000, 300000])
def test_calibrate_eq5_terms_on_rounding_ties(cuda_lib, T):
    """Eq. 5 terms placed on and next to the rounding ties of q = RNE(e 2^s).
    The kernel decides most terms in float32 and sends those within 2^-9 of a
    tie to its exact integer path; every field must still match the oracle
    bit for bit.  Exact ties: r = 1, |A| = 1, coef = (k + 1/2) 2^-s.  Near
    ties: coef = fl32((k + 1/2 + d) / (r |A| 2^s)) for d = +-3 2^-9 .. +-2^-22,
    which lands e 2^s within 2^-20 of its target.  The shift s is unchanged
    (these terms are far below max |e|)."""
    r_fp, r_bf, adv, mask, coef = (t.clone() for t in _inputs(T, 41))
    s = _ref(r_fp, r_bf, adv, mask, coef, 0.2, 0.2)["shift"]
    rng = np.random.default_rng(43)
    cand = np.nonzero((mask.numpy() != 0) & (adv.numpy() != 0))[0]
    pick = rng.choice(cand, size=max(64, T // 40), replace=False)
    rf, rb, a, c = r_fp.numpy(), r_bf.numpy(), adv.numpy(), coef.numpy()
    # the kernel's float32 path takes terms more than 2^-9 from a tie: 2^-8 and
    # 3 2^-9 land just outside that margin, the rest inside it
    deltas = [2.0 ** -9, -2.0 ** -9, 2.0 ** -10, -2.0 ** -10, 2.0 ** -12, -2.0 ** -12, 2.0 ** -22, -2.0 ** -22,
              2.0 ** -8, -2.0 ** -8, 3 * 2.0 ** -9, -3 * 2.0 ** -9]
    for j, i in enumerate(pick):
        k = int(rng.integers(0, 60))
        if j % 3 == 0:  # an exact tie on both ratios' terms
            rf[i] = rb[i] = 1.0
            a[i] = np.float32(1.0 if a[i] > 0 else -1.0)
            c[i] = np.float32(np.ldexp(k + 0.5, -s))
        else:  # near a tie, on the BF16 term (j odd) or the FP8 term (j even)
            r = float(rb[i] if j % 2 else rf[i])
            target = k + 0.5 + deltas[j % len(deltas)]
            c[i] = np.float32(target / (r * abs(float(a[i])) * 2.0 ** s))
    ref = _ref(r_fp, r_bf, adv, mask, coef, 0.2, 0.2)
    assert ref["shift"] == s
    # the planted terms do sit on or next to ties
    e = OC.update_terms(c[pick], rb[pick], a[pick])
    frac = np.abs(np.ldexp(np.abs(e), s) % 1.0 - 0.5)
    assert np.sum(frac == 0) >= len(pick) // 3 and np.sum(frac < 2.0 ** -8) >= len(pick) // 2
    got = _run(cuda_lib, r_fp, r_bf, adv, mask, coef, 0.2, 0.2)
    _compare(got, ref)
