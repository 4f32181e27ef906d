"""GPU parity: FP8 scoring with streaming logsumexp (a3/a4) and dense dlogits (a7).

Log-probs within 2e-3 absolute of the oracle's float64 log-softmax of its own
dequantised logits; ratios to the matching relative bound; dlogits within
2e-3 |g_t| per element.  Shapes span several 128x256 tiles, ragged T and V,
V = 1, T = 1, and the full configurations on 1024 random rows plus every
tile and band boundary.
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


def _data(T, H, V, seed, wstd=0.02):
    h = synth.normal_bf16(T, H, 1.0, seed, "cuda")
    W = synth.normal_bf16(V, H, wstd, seed + 1, "cuda")
    g = torch.Generator().manual_seed(seed)
    y = torch.randint(0, V, (T,), generator=g).to(torch.int32)
    y[0] = 0
    y[-1] = V - 1
    return h, W, y.cuda()


def _score(api, h, W, y, gran, logp_old=None):
    hc, hs = api.quantize(h, gran, api.ROLE_ACT)
    wc, ws = api.quantize(W, gran, api.ROLE_WEIGHT)
    out = api.token_logprobs(hc, hs, wc, ws, gran, y, logp_old)
    api.check()
    return out, (hc, hs, wc, ws)


@pytest.mark.parametrize("gran", [OQ.TENSOR, OQ.ROWWISE, OQ.BLOCK])
@pytest.mark.parametrize("T,H,V", [(1, 128, 1), (5, 128, 37), (300, 384, 1000), (257, 512, 4096),
                                   (130, 256, 513)])
def test_logprobs_small(cuda_lib, gran, T, H, V):
    h, W, y = _data(T, H, V, T * 7 + V)
    out, _ = _score(cuda_lib, h, W, y, gran)
    rows = np.arange(T)
    ref_lp, ref_lse, _ = oracle_logprobs_rows(h, W, gran, y, rows)
    assert np.max(np.abs(out["logp"].cpu().numpy() - ref_lp)) <= TOL
    assert np.max(np.abs(out["lse"].cpu().numpy() - ref_lse)) <= TOL


@pytest.mark.parametrize("gran", [OQ.TENSOR, OQ.ROWWISE])
def test_logprobs_hidden_not_multiple_of_128(cuda_lib, gran):
    h, W, y = _data(200, 208, 700, 3)
    out, _ = _score(cuda_lib, h, W, y, gran)
    ref_lp, _, _ = oracle_logprobs_rows(h, W, gran, y, np.arange(200))
    assert np.max(np.abs(out["logp"].cpu().numpy() - ref_lp)) <= TOL


def test_logprobs_tiny_grpo_full(cuda_lib):
    """The 2048 x 512 x 4096 per-tensor workload, every row, plus ratios."""
    w = synth.WORKLOADS["tiny_grpo"]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    logp_old = (torch.full((w.T,), -np.log(w.V)) + synth.old_policy_noise(w)).float().cuda()
    out, _ = _score(cuda_lib, h, W, y, w.gran, logp_old)
    ref_lp, _, _ = oracle_logprobs_rows(h, W, w.gran, y, np.arange(w.T))
    lp = out["logp"].cpu().numpy()
    assert np.max(np.abs(lp - ref_lp)) <= TOL
    ref_r = OL.importance_ratios(ref_lp, logp_old.cpu().numpy())
    assert np.max(np.abs(out["ratio"].cpu().numpy() / ref_r - 1)) <= 2.5e-3


def test_large_logits_stay_finite(cuda_lib):
    """Weights scaled so logits span +-100: the streaming logsumexp must not overflow."""
    h, W, y = _data(129, 256, 3000, 11, wstd=2.0)
    for gran in (OQ.TENSOR, OQ.BLOCK):
        out, _ = _score(cuda_lib, h, W, y, gran)
        ref_lp, _, _ = oracle_logprobs_rows(h, W, gran, y, np.arange(129))
        lp = out["logp"].cpu().numpy()
        assert np.all(np.isfinite(lp))
        assert np.max(np.abs(lp - ref_lp)) <= TOL * max(1.0, np.max(np.abs(ref_lp)) / 100)


@pytest.mark.parametrize("name,gran", [("grpo_8b", OQ.BLOCK), ("grpo_8b", OQ.TENSOR),
                                       ("grpo_8b", OQ.ROWWISE), ("dapo_32b", OQ.BLOCK),
                                       ("long_8b", OQ.BLOCK)])
def test_logprobs_full_size_sampled_rows(cuda_lib, name, gran):
    """Full configurations, in the launch configuration the bench uses: 1024
    random rows, both sides of every 128-row tile boundary and of every band
    boundary of the GEMM's tile order (64 token tiles), first and last rows."""
    w = synth.WORKLOADS[name]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    out, _ = _score(cuda_lib, h, W, y, gran)
    lp = out["logp"].cpu().numpy()
    assert np.all(np.isfinite(lp))
    rows = full_size_rows(w.T, 5)
    ref_lp, ref_lse, _ = oracle_logprobs_rows(h, W, gran, y, rows)
    assert np.max(np.abs(lp[rows] - ref_lp)) <= TOL
    assert np.max(np.abs(out["lse"].cpu().numpy()[rows] - ref_lse)) <= TOL


@pytest.mark.parametrize("gran", [OQ.TENSOR, OQ.BLOCK])
def test_dlogits_rows(cuda_lib, gran):
    T, H, V = 300, 256, 1100
    h, W, y = _data(T, H, V, 21)
    out, (hc, hs, wc, ws) = _score(cuda_lib, h, W, y, gran)
    g = (torch.randn(T, generator=torch.Generator().manual_seed(3)) * 1e-3).float().cuda()
    rows = torch.tensor([0, 5, 127, 128, 200, 299, 5], dtype=torch.int64, device="cuda")
    d = cuda_lib.dlogits_rows(hc, hs, wc, ws, gran, y, out["lse"], g, rows)
    cuda_lib.check()
    r = rows.cpu().numpy()
    _, ref_lse, z = oracle_logprobs_rows(h, W, gran, y, r)
    ref = OL.dlogits(z, y.cpu().numpy()[r], ref_lse, g.cpu().numpy()[r])
    gg = np.abs(g.cpu().numpy()[r])[:, None]
    assert np.all(np.abs(d.cpu().numpy() - ref) <= TOL * gg + 1e-12)
    # the one-hot column carries g (1 - p_y); the rows sum to ~0
    assert np.allclose(d.cpu().numpy().sum(1), 0, atol=1e-6)


def test_dlogits_tiny_grpo_all_rows(cuda_lib):
    w = synth.WORKLOADS["tiny_grpo"]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    out, (hc, hs, wc, ws) = _score(cuda_lib, h, W, y, w.gran)
    g = (torch.randn(w.T, generator=torch.Generator().manual_seed(4)) / w.T).float().cuda()
    rows = torch.arange(w.T, dtype=torch.int64, device="cuda")
    d = cuda_lib.dlogits_rows(hc, hs, wc, ws, w.gran, y, out["lse"], g, rows).cpu().numpy()
    cuda_lib.check()
    _, ref_lse, z = oracle_logprobs_rows(h, W, w.gran, y, np.arange(w.T))
    ref = OL.dlogits(z, y.cpu().numpy(), ref_lse, g.cpu().numpy())
    assert np.all(np.abs(d - ref) <= TOL * np.abs(g.cpu().numpy())[:, None] + 1e-12)


@pytest.mark.parametrize("gran", [OQ.BLOCK, OQ.TENSOR])
def test_logprobs_bit_reproducible_full_size(cuda_lib, gran):
    """No atomics on the scoring path: two calls on the grpo_8b batch give the
    same bits for logp, lse and the ratios."""
    w = synth.WORKLOADS["grpo_8b"]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    logp_old = (torch.full((w.T,), -12.0) + synth.old_policy_noise(w)).float().cuda()
    a, _ = _score(cuda_lib, h, W, y, gran, logp_old)
    b, _ = _score(cuda_lib, h, W, y, gran, logp_old)
    for k in ("logp", "lse", "ratio"):
        assert torch.equal(a[k], b[k]), k
