"""GPU parity: clipped surrogate, clip masks, counts and dloss/dlogp (a6/a7).

Clip masks and counts bit-exact; loss within 1e-4 relative (also against the
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
    for k in ("n_valid", "n_pos", "n_neg", "clipped_pos", "clipped_neg"):
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


def test_surrogate_deterministic(cuda_lib):
    r, adv, mask, w = (t.cuda() for t in _inputs(100000, 9))
    a = cuda_lib.read_clip_stats(cuda_lib.clipped_surrogate(r, adv, mask, w)["stats"])
    b = cuda_lib.read_clip_stats(cuda_lib.clipped_surrogate(r, adv, mask, w)["stats"])
    assert a["loss"] == b["loss"] and a["loss_sum"] == b["loss_sum"]
