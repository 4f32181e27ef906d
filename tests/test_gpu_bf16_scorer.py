"""GPU parity: the BF16 shadow-pass scorer (§4: reference ratios from BF16
forward passes), z = h W^T from the unquantised bf16 operands with fp32
accumulation on the tensor cores, streamed through the same logsumexp /
target-gather epilogue as the FP8 path.

Log-probs within 2e-3 absolute of the oracle's float64 log-softmax of the
float64 product of the same bf16 values (the workload statement's log-prob
tolerance); the observed error is far smaller because the products are exact
in fp32 and only the fp32 accumulation rounds.  Shapes span several 128 x 256
tiles, hidden sizes that are multiples of 64 but not of 128, ragged T and V,
strided rows, T = 1 and V = 1, and the full workloads on 1024 random rows
plus every tile and band boundary.
"""

import numpy as np
import pytest
import torch

from oracle import logprobs as OL
from paper_2609_22870_gb300 import synth
from tests.gpu_helpers import full_size_rows, oracle_bf16_logprobs_rows

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


def _oracle(h, W, y, rows):
    """Oracle (logp, lse) for the selected rows, one vocabulary strip of
    logits at a time (each z[t][v] is its own dot product)."""
    return oracle_bf16_logprobs_rows(h, W, y, rows)


@pytest.mark.parametrize("T,H,V", [(1, 64, 1), (5, 64, 37), (300, 192, 1000), (257, 512, 4096),
                                   (130, 128, 513), (129, 320, 2600)])
def test_bf16_logprobs_small(cuda_lib, T, H, V):
    h, W, y = _data(T, H, V, T * 11 + V)
    out = cuda_lib.bf16_token_logprobs(h, W, y)
    cuda_lib.check()
    ref_lp, ref_lse = _oracle(h, W, y, np.arange(T))
    assert np.max(np.abs(out["logp"].cpu().numpy() - ref_lp)) <= TOL
    assert np.max(np.abs(out["lse"].cpu().numpy() - ref_lse)) <= TOL


def test_bf16_strided_rows(cuda_lib):
    T, H, V = 200, 256, 900
    hw, Ww, y = _data(T, H + 64, V, 7)
    h, W = hw[:, 32:32 + H], Ww[:, 64:64 + H]  # row strides H + 64, 16-byte aligned starts
    out = cuda_lib.bf16_token_logprobs(h, W, y)
    cuda_lib.check()
    ref_lp, _ = _oracle(h.contiguous(), W.contiguous(), y, np.arange(T))
    assert np.max(np.abs(out["logp"].cpu().numpy() - ref_lp)) <= TOL


def test_bf16_tiny_grpo_all_rows_and_ratios(cuda_lib):
    w = synth.WORKLOADS["tiny_grpo"]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    logp_old = (torch.full((w.T,), -np.log(w.V)) + synth.old_policy_noise(w)).float().cuda()
    out = cuda_lib.bf16_token_logprobs(h, W, y, logp_old)
    cuda_lib.check()
    ref_lp, _ = _oracle(h, W, y, np.arange(w.T))
    lp = out["logp"].cpu().numpy()
    assert np.max(np.abs(lp - ref_lp)) <= TOL
    ref_r = OL.importance_ratios(ref_lp, logp_old.cpu().numpy())
    assert np.max(np.abs(out["ratio"].cpu().numpy() / ref_r - 1)) <= 2.5e-3


def test_bf16_large_logits_stay_finite(cuda_lib):
    h, W, y = _data(129, 256, 3000, 13, wstd=2.0)
    out = cuda_lib.bf16_token_logprobs(h, W, y)
    cuda_lib.check()
    ref_lp, _ = _oracle(h, W, y, np.arange(129))
    lp = out["logp"].cpu().numpy()
    assert np.all(np.isfinite(lp))
    assert np.max(np.abs(lp - ref_lp)) <= TOL * max(1.0, np.max(np.abs(ref_lp)) / 100)


@pytest.mark.parametrize("name", ["grpo_8b", "dapo_32b", "long_8b"])
def test_bf16_full_size_sampled_rows(cuda_lib, name):
    """1024 random rows, both sides of every 128-row tile boundary and of every
    band boundary of the tile order, first and last rows."""
    w = synth.WORKLOADS[name]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    out = cuda_lib.bf16_token_logprobs(h, W, y)
    cuda_lib.check()
    lp = out["logp"].cpu().numpy()
    assert np.all(np.isfinite(lp))
    rows = full_size_rows(w.T, 9)
    ref_lp, _ = _oracle(h, W, y, rows)
    assert np.max(np.abs(lp[rows] - ref_lp)) <= TOL


def test_bf16_rejects_bad_shapes_and_alignment(cuda_lib):
    h, W, y = _data(16, 128, 300, 3)
    with pytest.raises(cuda_lib.Fp8rlError) as e:
        cuda_lib.bf16_token_logprobs(h[:, :100], W[:, :100], y)
    assert e.value.status == cuda_lib.ESHAPE
    with pytest.raises(cuda_lib.Fp8rlError) as e:
        cuda_lib.bf16_token_logprobs(h[:, 4:68], W[:, 4:68], y)  # rows start 8 bytes in
    assert e.value.status == cuda_lib.EALIGN
    bad = y.clone()
    bad[3] = 300
    out = cuda_lib.bf16_token_logprobs(h, W, bad)
    assert cuda_lib.check_status() == cuda_lib.EDEVICE
    assert np.isnan(out["logp"].cpu().numpy()[3])
