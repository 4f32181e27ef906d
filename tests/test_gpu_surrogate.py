"""GPU parity: clipped surrogate, clip masks, counts and dloss/dlogp (a6/a7).

Clip masks, counts and clip fractions (computed by the library) bit-exact; loss within 1e-4 relative (also against the
mean |term|, the loss being a cancelling sum); gradient within 1e-6 relative.
"""

import numpy as np
import pytest
import torch

from oracle import surrogate as OS
from paper_2609_22870_gb300 import synth

pytestmark = pytest.mark.gpu


def _inputs(T, seed, ties=False):
    r_bf, r_fp, _ = synth.ratio_inputs(T, seed, sigma_old=0.2, sigma_fp8=0.1)
    g = torch.Generator().manual_seed(seed)
    adv = torch.randn(T, generator=g).float()
    adv[torch.rand(T, generator=g) < 0.05] = 0
    mask = (torch.rand(T, generator=g) < 0.85).to(torch.uint8)
    w = torch.rand(T, generator=g).float() * 2
    if ties:  # ratios exactly at the bounds
        r_fp[::5] = 0.8
        r_fp[1::5] = 1.2
    return r_fp, adv, mask, w


def _check(api, r, adv, mask, w, lo, hi, bounds=None):
    d = [None if t is None else t.cuda() for t in (r, adv, mask, w)]
    out = api.clipped_surrogate(*d, lo=lo, hi=hi, bounds=bounds)
    api.check()
    st = api.read_clip_stats(out["stats"])
    L, H = (float(bounds[0]), float(bounds[1])) if bounds is not None else (lo, hi)
    ref = OS.clipped_surrogate(r.numpy(), adv.numpy(), None if mask is None else mask.numpy(),
                               None if w is None else w.numpy(), L, H)
    assert np.array_equal(out["clip_mask"].cpu().numpy(), ref["clip_mask"])
    for k in ("n_valid", "n_pos", "n_neg", "clipped_pos", "clipped_neg", "clip_frac_pos", "clip_frac_neg",
              "clip_frac"):
        assert st[k] == ref[k], k
    scale = max(abs(ref["loss"]), np.sum(np.abs(ref["terms"])) / max(1, ref["n_valid"]), 1e-300)
    assert abs(st["loss"] - ref["loss"]) <= 1e-4 * abs(ref["loss"]) + 1e-12 * scale
    assert abs(st["loss"] - ref["loss"]) <= 1e-4 * scale
    g = out["grad"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(g - ref["grad"]) <= 1e-6 * np.abs(ref["grad"]) + 1e-30)
    assert np.all(g[ref["grad"] == 0] == 0)
    return st


@pytest.mark.parametrize("T", [1, 31, 1000, 16384, 131072])
@pytest.mark.parametrize("bounds", [(0.8, 1.2), (0.6, 1.8), (0.83, 1.27)])
def test_surrogate_parity(cuda_lib, T, bounds):
    _check(cuda_lib, *_inputs(T, T), *bounds)


def test_surrogate_bounds_from_device_and_ties(cuda_lib):
    r, adv, mask, w = _inputs(5000, 3, ties=True)
    b = torch.tensor([0.8, 1.2], dtype=torch.float32, device="cuda")
    st = _check(cuda_lib, r, adv, mask, w, 0.1, 9.0, bounds=b)
    assert st["lo"] == np.float32(0.8) and st["hi"] == np.float32(1.2)


def test_surrogate_nullable_and_empty(cuda_lib):
    r, adv, _, _ = _inputs(777, 4)
    _check(cuda_lib, r, adv, None, None, 0.8, 1.2)
    st = _check(cuda_lib, r, adv, torch.zeros(777, dtype=torch.uint8), None, 0.8, 1.2)
    assert st["loss"] == 0 and st["flags"] == 1


def test_surrogate_with_the_calibrations_valid_count(cuda_lib):
    """The step passes the calibration's count of valid tokens (same mask), so
    the surrogate skips its counting pass: results identical to the counting
    call.  A count of twice the valid tokens halves the gradient and the loss
    exactly (the pointer is read); without a mask it is ignored."""
    api = cuda_lib
    T = 70000
    r, adv, mask, w = (t.cuda() for t in _inputs(T, 21))
    r_bf = (r * 1.01).contiguous()
    cal = api.calibrate_clip_bounds(r, r_bf, adv, mask, None, 0.2, 0.2)
    nv = api.n_valid_view(cal)
    assert int(nv.item()) == int(mask.sum().item()) == api.read_calib_result(cal)["n_valid"]
    b = api.bounds_view(cal)
    ref = api.clipped_surrogate(r, adv, mask, w, bounds=b)
    got = api.clipped_surrogate(r, adv, mask, w, bounds=b, n_valid=nv)
    api.check()
    assert torch.equal(ref["grad"], got["grad"]) and torch.equal(ref["clip_mask"], got["clip_mask"])
    assert api.read_clip_stats(ref["stats"]) == api.read_clip_stats(got["stats"])
    twice = (2 * nv).contiguous()
    half = api.clipped_surrogate(r, adv, mask, w, bounds=b, n_valid=twice)
    api.check()
    assert torch.equal(half["grad"] * 2, ref["grad"])
    assert api.read_clip_stats(half["stats"])["loss"] * 2 == api.read_clip_stats(ref["stats"])["loss"]
    nomask = api.clipped_surrogate(r, adv, None, w, bounds=b, n_valid=twice)
    api.check()
    assert api.read_clip_stats(nomask["stats"])["n_valid"] == T


def test_surrogate_deterministic(cuda_lib):
    r, adv, mask, w = (t.cuda() for t in _inputs(100000, 9))
    a = cuda_lib.read_clip_stats(cuda_lib.clipped_surrogate(r, adv, mask, w)["stats"])
    b = cuda_lib.read_clip_stats(cuda_lib.clipped_surrogate(r, adv, mask, w)["stats"])
    assert a["loss"] == b["loss"] and a["loss_sum"] == b["loss_sum"]


# ---- sequence-mean variant ---------------------------------------------------

def _seq_ids(T, n_seq, seed, contiguous=True):
    g = torch.Generator().manual_seed(seed + 7)
    if contiguous:  # packed responses of random lengths
        cuts = torch.sort(torch.randint(0, T + 1, (n_seq - 1,), generator=g)).values
        sid = torch.bucketize(torch.arange(T), cuts, right=True)
    else:
        sid = torch.randint(0, n_seq, (T,), generator=g)
    return sid.to(torch.int32)


def _check_seq(api, r, adv, mask, w, sid, n_seq, lo, hi):
    d = [None if t is None else t.cuda() for t in (r, adv, sid, mask, w)]
    out = api.clipped_surrogate_seq_mean(d[0], d[1], d[2], n_seq, mask=d[3], w_tis=d[4], lo=lo, hi=hi)
    api.check()
    st = api.read_clip_stats(out["stats"])
    ref = OS.clipped_surrogate_seq_mean(r.numpy(), adv.numpy(), None if mask is None else mask.numpy(),
                                        None if w is None else w.numpy(), lo, hi, sid.numpy(), n_seq)
    assert np.array_equal(out["clip_mask"].cpu().numpy(), ref["clip_mask"])
    for k in ("n_valid", "n_pos", "n_neg", "clipped_pos", "clipped_neg", "n_seq_valid", "clip_frac_pos",
              "clip_frac_neg", "clip_frac"):
        assert st[k] == ref[k], k
    n = max(1, ref["n_valid"])
    scale = max(abs(ref["loss"]), np.sum(np.abs(ref["terms"])) / n, 1e-300)
    assert abs(st["loss"] - ref["loss"]) <= 1e-4 * scale
    g = out["grad"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(g - ref["grad"]) <= 1e-6 * np.abs(ref["grad"]) + 1e-30)
    assert np.all(g[ref["grad"] == 0] == 0)
    return st


@pytest.mark.parametrize("T,n_seq", [(1, 1), (100, 7), (5000, 32), (65536, 128), (131072, 8)])
@pytest.mark.parametrize("contiguous", [True, False])
def test_seq_mean_parity(cuda_lib, T, n_seq, contiguous):
    r, adv, mask, w = _inputs(T, T + n_seq)
    _check_seq(cuda_lib, r, adv, mask, w, _seq_ids(T, n_seq, T, contiguous), n_seq, 0.8, 1.2)


def test_seq_mean_equal_lengths_match_token_mean_and_empty(cuda_lib):
    T, n_seq = 4096, 8
    r, adv, _, w = _inputs(T, 5)
    sid = torch.arange(T, dtype=torch.int32) // (T // n_seq)
    st = _check_seq(cuda_lib, r, adv, None, w, sid, n_seq, 0.8, 1.2)
    tok = cuda_lib.read_clip_stats(cuda_lib.clipped_surrogate(r.cuda(), adv.cuda(), None, w.cuda())["stats"])
    assert abs(st["loss"] - tok["loss"]) <= 1e-5 * max(abs(tok["loss"]), 1e-6)
    st0 = _check_seq(cuda_lib, r, adv, torch.zeros(T, dtype=torch.uint8), w, sid, n_seq + 3, 0.8, 1.2)
    assert st0["loss"] == 0 and st0["n_seq_valid"] == 0 and st0["flags"] == 1


def test_seq_mean_bad_ids_flagged(cuda_lib):
    r, adv, mask, w = (t.cuda() for t in _inputs(300, 6))
    sid = torch.zeros(300, dtype=torch.int32, device="cuda")
    sid[17] = 5  # n_seq = 5: out of range
    cuda_lib.clipped_surrogate_seq_mean(r, adv, sid, 5, mask=mask, w_tis=w)
    assert cuda_lib.check_status() == cuda_lib.EDEVICE
