"""GPU parity: §3 diagnostics (over-clipping, clip counts, probability and
ratio NMAE against BF16 references) and the §2.3 TIS weight.

Counts bit-exact (the same float32 comparisons on the same inputs); ratio NMAE
within 1e-6 relative (the differences of float32 ratios within a factor of two
are exact, only the summation rounds); probability NMAE within 1e-5 relative
(|p8 - pb| is formed as pb |expm1(l8 - lb)| from an exact float32 difference,
so the error is a few float32 roundings of expf / expm1f); TIS weights within
2e-6 relative (expf of a rounded float32 difference, then min with C).  Sizes
span several blocks and a ragged tail, unaligned (scalar-path) inputs, no
mask, no log-probs, T = 0, and the 8B workload's full batch.
"""

import numpy as np
import pytest
import torch

from oracle import diagnostics as OD
from paper_2609_22870_gb300 import synth

pytestmark = pytest.mark.gpu


def _inputs(T, seed, ties=False):
    g = torch.Generator().manual_seed(seed)
    lb = (torch.randn(T, generator=g) * 2 - 8).float()
    l8 = (lb + torch.randn(T, generator=g) * 0.02).float()
    lold = (lb + torch.randn(T, generator=g) * 0.05).float()
    rb = torch.exp(lb - lold).float()
    r8 = torch.exp(l8 - lold).float()
    if ties:  # ratios exactly on the bounds
        idx = torch.randint(0, T, (T // 10,), generator=g)
        r8[idx[: len(idx) // 2]] = float(np.float32(0.8))
        rb[idx[len(idx) // 2:]] = float(np.float32(1.2))
    A = torch.randn(T, generator=g).float()
    A[torch.rand(T, generator=g) < 0.05] = 0.0
    m = (torch.rand(T, generator=g) < 0.85).to(torch.uint8)
    return l8, lb, r8, rb, A, m


def _check(api, l8, lb, r8, rb, A, m, eps_lo, eps_hi, with_p=True, with_mask=True):
    dev = lambda t: None if t is None else t.cuda()  # noqa: E731
    buf = api.clip_diagnostics(dev(r8), dev(rb), dev(A), dev(m) if with_mask else None,
                               dev(l8) if with_p else None, dev(lb) if with_p else None, eps_lo, eps_hi)
    api.check()
    got = api.read_clip_diag(buf)
    ref = OD.clip_diagnostics(l8.numpy() if with_p else None, lb.numpy() if with_p else None, r8.numpy(),
                              rb.numpy(), A.numpy(), m.numpy() if with_mask else None, eps_lo, eps_hi)
    for k in ("n_valid", "n_pos", "n_neg", "clipped_lo_fp8", "clipped_hi_fp8", "clipped_lo_bf16",
              "clipped_hi_bf16", "over_clipped_lo", "over_clipped_hi"):
        assert got[k] == ref[k], (k, got[k], ref[k])
    assert np.float32(got["c_lo"]) == ref["c_lo"] and np.float32(got["c_hi"]) == ref["c_hi"]
    if ref["n_valid"]:
        assert abs(got["nmae_ratio"] / ref["nmae_ratio"] - 1) <= 1e-6
        if with_p:
            assert abs(got["nmae_prob"] / ref["nmae_prob"] - 1) <= 1e-5
        else:
            assert np.isnan(got["nmae_prob"]) and got["flags"] & 2
    return got, ref


@pytest.mark.parametrize("T", [1, 7, 1000, 4099, 262147])
def test_diagnostics_match_oracle(cuda_lib, T):
    _check(cuda_lib, *_inputs(T, T), 0.2, 0.28)


def test_diagnostics_ties_no_mask_no_logprobs(cuda_lib):
    x = _inputs(50000, 3, ties=True)
    got, ref = _check(cuda_lib, *x, 0.2, 0.2, with_p=True, with_mask=False)
    assert ref["over_clipped_lo"] > 0 and ref["over_clipped_hi"] >= 0
    _check(cuda_lib, *x, 0.2, 0.2, with_p=False, with_mask=True)


def test_diagnostics_unaligned_scalar_path(cuda_lib):
    l8, lb, r8, rb, A, m = _inputs(10001, 5)
    dv = lambda t: t.cuda()[1:]  # noqa: E731  (4 bytes past a 16-byte boundary)
    buf = cuda_lib.clip_diagnostics(dv(r8), dv(rb), dv(A), dv(m), dv(l8), dv(lb), 0.2, 0.2)
    cuda_lib.check()
    got = cuda_lib.read_clip_diag(buf)
    ref = OD.clip_diagnostics(l8[1:].numpy(), lb[1:].numpy(), r8[1:].numpy(), rb[1:].numpy(),
                              A[1:].numpy(), m[1:].numpy(), 0.2, 0.2)
    assert got["over_clipped_lo"] == ref["over_clipped_lo"]
    assert got["clipped_hi_fp8"] == ref["clipped_hi_fp8"]
    assert abs(got["nmae_prob"] / ref["nmae_prob"] - 1) <= 1e-5


def test_diagnostics_empty(cuda_lib):
    e = torch.empty(0, device="cuda")
    got = cuda_lib.read_clip_diag(cuda_lib.clip_diagnostics(e, e, e))
    cuda_lib.check()
    assert got["n_valid"] == 0 and got["flags"] & 1 and np.isnan(got["nmae_ratio"])


def test_diagnostics_full_8b_batch(cuda_lib):
    w = synth.WORKLOADS["grpo_8b"]
    adv, mask = synth.rollout(w)
    l8, lb, r8, rb, _, _ = _inputs(w.T, 11)
    _check(cuda_lib, l8, lb, r8, rb, adv, mask, w.eps_low, w.eps_high)


@pytest.mark.parametrize("T", [1, 5000, 300001])
def test_tis_weights(cuda_lib, T):
    g = torch.Generator().manual_seed(T)
    lo = (torch.randn(T, generator=g) * 3 - 5).float()
    ls = (lo + torch.randn(T, generator=g)).float()
    w = cuda_lib.tis_weights(lo.cuda(), ls.cuda(), 2.0).cpu().numpy()
    cuda_lib.check()
    ref = OD.tis_weights(lo.numpy(), ls.numpy(), 2.0)
    assert np.all(w <= 2.0)
    assert np.max(np.abs(w / ref - 1)) <= 2e-6
    assert np.all(w[ref >= 2.0] == 2.0)
