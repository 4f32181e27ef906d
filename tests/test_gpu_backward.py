"""GPU parity: backward through the FP8 lm_head (dh = P W, dW = P^T h with
P = dLoss/dlogits recomputed from the FP8 logits).

Tolerance from the arithmetic: the kernel rounds each P[t][v] to bf16
(relative 2^-9) and accumulates in float32, so each output element is within
2^-8 of the sum of the absolute values of its terms, sum_v |P[t][v] W[v][k]|
(for dh) or sum_t |P[t][v] h[t][k]| (for dW), which the oracle computes from
its own float64 P.  Small shapes compare every element; the full grpo_8b shape
compares sampled rows of dh and checks that every column of dW sums to ~0
(each row of P sums to g_t (1 - 1) = 0).
"""

import numpy as np
import pytest
import torch

from oracle import logprobs as OL
from oracle import quantize as OQ
from paper_2609_22870_gb300 import synth
from tests.gpu_helpers import STRIP, oracle_logprobs_rows, sample_rows

pytestmark = pytest.mark.gpu
REL = 2.0 ** -8


def _data(T, H, V, seed, wstd=0.05):
    h = synth.normal_bf16(T, H, 1.0, seed, "cuda")
    W = synth.normal_bf16(V, H, wstd, seed + 1, "cuda")
    g = torch.Generator().manual_seed(seed)
    y = torch.randint(0, V, (T,), generator=g).to(torch.int32)
    y[0] = 0
    y[-1] = V - 1
    gl = (torch.randn(T, generator=g) / T).float()
    gl[::11] = 0  # masked tokens
    return h, W, y.cuda(), gl.cuda()


def _forward_backward(api, h, W, y, g, gran, **kw):
    hc, hs = api.quantize(h, gran, api.ROLE_ACT)
    wc, ws = api.quantize(W, gran, api.ROLE_WEIGHT)
    fwd = api.token_logprobs(hc, hs, wc, ws, gran, y)
    out = api.lm_head_backward(hc, hs, wc, ws, gran, y, fwd["lse"], g, h, W, **kw)
    api.check()
    return out, (hc, hs, wc, ws, fwd["lse"])


def _oracle(h, W, y, g, gran):
    h32, W32 = h.float().cpu().numpy(), W.float().cpu().numpy()
    hq, hs = OQ.quantize(h32, gran, OQ.ACT)
    wq, ws = OQ.quantize(W32, gran, OQ.WEIGHT)
    ref = OL.lm_head_backward(hq, hs, wq, ws, gran, y.cpu().numpy(), g.cpu().numpy(), h32, W32)
    aP = np.abs(ref["P"])
    return ref, aP @ np.abs(W32.astype(np.float64)), aP.T @ np.abs(h32.astype(np.float64))


@pytest.mark.parametrize("gran", [OQ.TENSOR, OQ.ROWWISE, OQ.BLOCK])
@pytest.mark.parametrize("T,H,V", [(300, 256, 1000), (129, 384, 1001), (1, 128, 1), (520, 128, 4096)])
def test_backward_small_all_elements(cuda_lib, gran, T, H, V):
    h, W, y, g = _data(T, H, V, T + V)
    out, _ = _forward_backward(cuda_lib, h, W, y, g, gran)
    ref, bh, bw = _oracle(h, W, y, g, gran)
    dh = out["dh"].cpu().numpy().astype(np.float64)
    dW = out["dW"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(dh - ref["dh"]) <= REL * bh + 1e-30)
    assert np.all(np.abs(dW - ref["dW"]) <= REL * bw + 1e-30)
    assert np.all(dh[g.cpu().numpy() == 0] == 0)  # g = 0 rows: P is exactly 0


def test_backward_accumulate_chunks_and_single_outputs(cuda_lib):
    api = cuda_lib
    T, H, V, gran = 512, 256, 2048, OQ.BLOCK
    h, W, y, g = _data(T, H, V, 5)
    full, (hc, hs, wc, ws, lse) = _forward_backward(api, h, W, y, g, gran)
    # the same call twice into one dW with accumulation: exactly twice (deterministic GEMM)
    dW = full["dW"].clone()
    api.lm_head_backward(hc, hs, wc, ws, gran, y, lse, g, h, W, want_dh=False, accumulate_dw=True,
                         out={"dW": dW})
    api.check()
    assert torch.equal(dW, 2 * full["dW"])
    # two token chunks accumulated = the whole batch (different summation order)
    acc = torch.zeros_like(full["dW"])
    for t0, t1 in ((0, 256), (256, 512)):
        hc_c, hs_c = api.quantize(h[t0:t1].contiguous(), gran, api.ROLE_ACT)
        api.lm_head_backward(hc_c, hs_c, wc, ws, gran, y[t0:t1].contiguous(), lse[t0:t1].contiguous(),
                             g[t0:t1].contiguous(), h[t0:t1].contiguous(), W, want_dh=False,
                             accumulate_dw=True, out={"dW": acc})
    api.check()
    scale = full["dW"].abs().max().item()
    assert (acc - full["dW"]).abs().max().item() <= 1e-5 * scale
    only_dh = api.lm_head_backward(hc, hs, wc, ws, gran, y, lse, g, h, W, want_dw=False)
    api.check()
    assert only_dh["dW"] is None and torch.equal(only_dh["dh"], full["dh"])
    with pytest.raises(RuntimeError):
        api.lm_head_backward(hc, hs, wc, ws, gran, y, lse, g, h, W, want_dh=False, want_dw=False)


@pytest.mark.parametrize("gran", [OQ.BLOCK, OQ.TENSOR])
def test_backward_full_size_grpo8b(cuda_lib, gran):
    """grpo_8b (T 16384, H 4096, V 151936): sampled rows of dh against the
    oracle; dW by its zero column sums."""
    api = cuda_lib
    w = synth.WORKLOADS["grpo_8b"]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    g = (torch.randn(w.T, generator=torch.Generator().manual_seed(8)) / w.T).float().cuda()
    out, _ = _forward_backward(api, h, W, y, g, gran)
    dh = out["dh"]
    assert bool(torch.isfinite(dh).all()) and bool(torch.isfinite(out["dW"]).all())
    rows = sample_rows(w.T, 6, 9)
    _, lse_r, z_r = oracle_logprobs_rows(h, W, gran, y, rows)
    P = OL.dlogits(z_r, y.cpu().numpy()[rows], lse_r, g.cpu().numpy()[rows])
    ref = np.zeros((len(rows), w.H))
    bound = np.zeros((len(rows), w.H))
    for v0 in range(0, w.V, STRIP):
        Ws = W[v0:v0 + STRIP].float().cpu().numpy().astype(np.float64)
        ref += P[:, v0:v0 + STRIP] @ Ws
        bound += np.abs(P[:, v0:v0 + STRIP]) @ np.abs(Ws)
    got = dh[torch.as_tensor(rows, device="cuda")].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - ref) <= REL * bound + 1e-30)
    # columns of dW: sum_v dW[v][k] = sum_t (sum_v P[t][v]) h[t][k], and each
    # row of the bf16 P sums to within 2^-8 |g_t| of 0
    col = out["dW"].double().sum(0)
    lim = REL * (g.abs().double()[:, None] * h.double().abs()).sum(0)
    assert bool((col.abs() <= lim + 1e-6 * out["dW"].abs().double().sum(0)).all())
