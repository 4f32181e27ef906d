"""Pins for the oracle's §3 diagnostics and the §2.3 TIS weight.

A hand-worked table (tests/golden/diagnostics_tiny.txt) that hits every case
of the over-clipping definitions, the equality conventions, A = 0 and the mask;
set identities between the clip and over-clip counts on random inputs; closed
forms of NMAE; the identity inputs (FP8 == BF16) giving no over-clipping and
zero error; and closed forms of the truncated importance weight.
"""

import os

import numpy as np
import pytest

from oracle import diagnostics as D

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _table():
    rows = []
    for line in open(os.path.join(GOLDEN, "diagnostics_tiny.txt")):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        rows.append((float(f[0]), float(f[1]), float(f[2]), int(f[3])))
    return [np.array(c) for c in zip(*rows)]


def test_hand_worked_table():
    r8, rb, A, m = _table()
    d = D.clip_diagnostics(None, None, r8, rb, A, m, 0.2, 0.2)
    assert (d["n_valid"], d["n_pos"], d["n_neg"]) == (7, 3, 3)
    assert (d["clipped_lo_fp8"], d["clipped_hi_fp8"]) == (2, 2)
    assert (d["clipped_lo_bf16"], d["clipped_hi_bf16"]) == (1, 2)
    assert (d["over_clipped_lo"], d["over_clipped_hi"]) == (1, 1)
    # decimal hand sums of float32 inputs: agreement to float32 input precision
    assert abs(d["nmae_ratio"] - 0.65 / 6.7) < 1e-6
    assert np.isnan(d["nmae_prob"])


def test_identity_inputs_have_no_over_clipping():
    rng = np.random.default_rng(0)
    T = 5000
    r = np.exp(rng.normal(0, 0.2, T)).astype(np.float32)
    A = rng.normal(0, 1, T).astype(np.float32)
    lp = (rng.normal(-3, 1, T)).astype(np.float32)
    m = (rng.random(T) < 0.9).astype(np.uint8)
    d = D.clip_diagnostics(lp, lp, r, r, A, m, 0.2, 0.28)
    assert d["over_clipped_lo"] == 0 and d["over_clipped_hi"] == 0
    assert d["clipped_lo_fp8"] == d["clipped_lo_bf16"] > 0
    assert d["clipped_hi_fp8"] == d["clipped_hi_bf16"] > 0
    assert d["nmae_ratio"] == 0.0 and d["nmae_prob"] == 0.0


def test_set_identities_on_random_inputs():
    # clipped_fp8 - clipped_bf16 = over - under (per bound), with `under` the
    # mirror-image count; and over-clipped tokens are a subset of FP8-clipped
    rng = np.random.default_rng(1)
    T = 20000
    rb = np.exp(rng.normal(0, 0.15, T)).astype(np.float32)
    r8 = (rb * np.exp(rng.normal(0, 0.08, T))).astype(np.float32)
    A = np.round(rng.normal(0, 1, T), 1).astype(np.float32)  # some exact zeros
    m = (rng.random(T) < 0.8).astype(np.uint8)
    d = D.clip_diagnostics(None, None, r8, rb, A, m, 0.2, 0.2)
    under = D.clip_diagnostics(None, None, rb, r8, A, m, 0.2, 0.2)  # roles swapped
    assert d["clipped_lo_fp8"] - d["clipped_lo_bf16"] == d["over_clipped_lo"] - under["over_clipped_lo"]
    assert d["clipped_hi_fp8"] - d["clipped_hi_bf16"] == d["over_clipped_hi"] - under["over_clipped_hi"]
    assert 0 < d["over_clipped_lo"] <= d["clipped_lo_fp8"]
    assert 0 < d["over_clipped_hi"] <= d["clipped_hi_fp8"]
    assert d["n_pos"] + d["n_neg"] + int(((A == 0) & (m != 0)).sum()) == d["n_valid"]


def test_nmae_closed_forms():
    ref = np.array([1.0, 2.0, 4.0])
    assert D.nmae(ref, ref) == 0.0
    assert np.isclose(D.nmae(ref * 1.25, ref), 0.25, rtol=0, atol=1e-15)
    x = np.array([1.5, 1.0, 5.0])
    assert np.isclose(D.nmae(7 * x, 7 * ref), D.nmae(x, ref), rtol=1e-15)  # scale invariance
    assert np.isclose(D.nmae([2.0, 2.0, 4.0], ref), 1.0 / 7.0, rtol=0, atol=1e-15)
    assert np.isnan(D.nmae([1.0], [0.0]))


def test_probability_nmae_is_exp_of_logprobs():
    lp_b = np.log(np.array([0.5, 0.25], np.float32))
    lp_8 = np.log(np.array([0.25, 0.25], np.float32))
    d = D.clip_diagnostics(lp_8, lp_b, np.ones(2, np.float32), np.ones(2, np.float32),
                           np.ones(2, np.float32), None, 0.2, 0.2)
    assert np.isclose(d["nmae_prob"], 0.25 / 0.75, rtol=1e-7)


@pytest.mark.parametrize("C", [2.0, 1.5])
def test_tis_weight_closed_forms(C):
    lo = np.float32([-3.0, -2.0, -2.0, -10.0])
    ls = np.float32([-3.0, -2.0 - np.log(3.0), -2.0 + np.log(2.0), -10.0 + np.log(4.0)])
    w = D.tis_weights(lo, ls, C)
    assert w[0] == 1.0
    assert w[1] == C  # ratio 3 truncated
    assert abs(w[2] - 0.5) < 1e-6
    assert abs(w[3] - 0.25) < 1e-6
    assert np.all(w <= C)
