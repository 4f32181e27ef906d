"""GPU parity: scoring with power-of-two (UE8M0) block scales applied by the
tensor cores' block-scaled MMA (tcgen05.mma kind::mxf8f6f4, E8M0 scale
factors in TMEM), FP8RL_GRAN_BLOCK_UE8M0.

The codes and scales are those of fp8rl_quantize_ue8m0 at block granularity
(bit-exact against the oracle in test_gpu_quantize.py).  Log-probs within the
workload's 2e-3 of the oracle's float64 log-softmax of its own power-of-two
quantisation; against the register-promotion path (FP8RL_GRAN_BLOCK) on the
same codes the logits differ only in float32 summation order, so the log-probs
agree to 1e-5.  A scale that is not a power of two is bad input.
"""

import numpy as np
import pytest
import torch

from oracle import logprobs as OL
from oracle import quantize as OQ
from paper_2609_22870_gb300 import synth
from tests.gpu_helpers import full_size_rows, oracle_logprobs_rows

pytestmark = pytest.mark.gpu
TOL = 2e-3
UE = 3  # FP8RL_GRAN_BLOCK_UE8M0


def _data(T, H, V, seed, wstd=0.05):
    h = synth.normal_bf16(T, H, 1.0, seed, "cuda")
    W = synth.normal_bf16(V, H, wstd, seed + 1, "cuda")
    g = torch.Generator().manual_seed(seed)
    y = torch.randint(0, V, (T,), generator=g).to(torch.int32)
    y[0] = 0
    y[-1] = V - 1
    return h, W, y.cuda()


def _codes(api, h, W):
    hc, hs = api.quantize(h, api.GRAN_BLOCK, api.ROLE_ACT, ue8m0=True)
    wc, ws = api.quantize(W, api.GRAN_BLOCK, api.ROLE_WEIGHT, ue8m0=True)
    return hc, hs, wc, ws


@pytest.mark.parametrize("T,H,V", [(1, 128, 1), (5, 128, 37), (300, 384, 1000), (257, 512, 4096),
                                   (130, 256, 513), (700, 1024, 3000)])
def test_ue8m0_mma_small(cuda_lib, T, H, V):
    api = cuda_lib
    h, W, y = _data(T, H, V, T * 3 + V)
    hc, hs, wc, ws = _codes(api, h, W)
    out = api.token_logprobs(hc, hs, wc, ws, UE, y)
    api.check()
    ref_lp, ref_lse, _ = oracle_logprobs_rows(h, W, OQ.BLOCK, y, np.arange(T), pow2=True)
    assert np.max(np.abs(out["logp"].cpu().numpy() - ref_lp)) <= TOL
    assert np.max(np.abs(out["lse"].cpu().numpy() - ref_lse)) <= TOL
    # the promotion path on the same codes: same exact products, other order
    prom = api.token_logprobs(hc, hs, wc, ws, api.GRAN_BLOCK, y)
    api.check()
    assert (out["logp"] - prom["logp"]).abs().max().item() <= 1e-5
    assert (out["lse"] - prom["lse"]).abs().max().item() <= 1e-5


@pytest.mark.parametrize("name", ["grpo_8b", "dapo_32b"])
def test_ue8m0_mma_full_size(cuda_lib, name):
    """Full workloads in the bench's launch configuration: 1024 random rows,
    both sides of every tile and band boundary, first and last rows."""
    api = cuda_lib
    w = synth.WORKLOADS[name]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    hc, hs, wc, ws = _codes(api, h, W)
    out = api.token_logprobs(hc, hs, wc, ws, UE, y)
    api.check()
    lp = out["logp"].cpu().numpy()
    assert np.all(np.isfinite(lp))
    rows = full_size_rows(w.T, 13)
    ref_lp, _, _ = oracle_logprobs_rows(h, W, OQ.BLOCK, y, rows, pow2=True)
    assert np.max(np.abs(lp[rows] - ref_lp)) <= TOL


def test_ue8m0_mma_bit_reproducible(cuda_lib):
    api = cuda_lib
    h, W, y = _data(1024, 512, 5000, 91)
    hc, hs, wc, ws = _codes(api, h, W)
    a = api.token_logprobs(hc, hs, wc, ws, UE, y)
    b = api.token_logprobs(hc, hs, wc, ws, UE, y)
    api.check()
    assert torch.equal(a["logp"], b["logp"]) and torch.equal(a["lse"], b["lse"])


def test_ue8m0_mma_dlogits_rows(cuda_lib):
    """Dense dlogits rows run on the hardware-scaled recompute too (the
    variant's backward is checked against the oracle with the other backward
    tests)."""
    api = cuda_lib
    T, H, V = 300, 256, 1100
    h, W, y = _data(T, H, V, 93)
    hc, hs, wc, ws = _codes(api, h, W)
    fwd = api.token_logprobs(hc, hs, wc, ws, UE, y)
    g = (torch.randn(T, generator=torch.Generator().manual_seed(94)) * 1e-3).float().cuda()
    rows = torch.tensor([0, 5, 127, 128, 200, 299], dtype=torch.int64, device="cuda")
    d = api.dlogits_rows(hc, hs, wc, ws, UE, y, fwd["lse"], g, rows)
    api.check()
    r = rows.cpu().numpy()
    _, ref_lse, z = oracle_logprobs_rows(h, W, OQ.BLOCK, y, r, pow2=True)
    ref = OL.dlogits(z, y.cpu().numpy()[r], ref_lse, g.cpu().numpy()[r])
    gg = np.abs(g.cpu().numpy()[r])[:, None]
    assert np.all(np.abs(d.cpu().numpy() - ref) <= TOL * gg + 1e-12)


def test_ue8m0_mma_rejects_scales_that_are_not_powers_of_two(cuda_lib):
    api = cuda_lib
    h, W, y = _data(200, 256, 700, 95)
    hc, hs = api.quantize(h, api.GRAN_BLOCK, api.ROLE_ACT)          # the paper's amax / 448 scales
    wc, ws = api.quantize(W, api.GRAN_BLOCK, api.ROLE_WEIGHT, ue8m0=True)
    api.token_logprobs(hc, hs, wc, ws, UE, y)
    assert api.check_status() == api.EDEVICE
    api.check()


def test_ue8m0_mma_step_through_the_binding(cuda_lib):
    """score_calibrate_loss with the UE8M0 granularity: the binding quantises
    with power-of-two block scales and the scoring runs on the block-scaled
    MMA; log-probs against the oracle's power-of-two path."""
    api = cuda_lib
    T, H, V = 640, 512, 3000
    h, W, y = _data(T, H, V, 97)
    g = torch.Generator().manual_seed(98)
    logp_old = (torch.randn(T, generator=g) * 0.01 - 8.0).float().cuda()
    r_bf16 = torch.exp(torch.randn(T, generator=g) * 0.01).float().cuda()
    adv = torch.randn(T, generator=g).float().cuda()
    mask = torch.ones(T, dtype=torch.uint8, device="cuda")
    coef = torch.ones(T, dtype=torch.float32, device="cuda")
    b = api.score_calibrate_loss(h, W, y, logp_old, r_bf16, adv, mask, coef, UE, 0.2, 0.2)
    api.check()
    ref_lp, _, _ = oracle_logprobs_rows(h, W, OQ.BLOCK, y, np.arange(T), pow2=True)
    assert np.max(np.abs(b.logp.cpu().numpy() - ref_lp)) <= TOL
    hc, hs = api.quantize(h, api.GRAN_BLOCK, api.ROLE_ACT, ue8m0=True)
    assert torch.equal(b.h_codes, hc) and torch.equal(b.h_scales[:hs.numel()], hs)
