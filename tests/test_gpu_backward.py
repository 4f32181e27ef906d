"""GPU parity: the FP8 backward through the lm_head (dh = P W, dW = P^T h,
P = dLoss/dlogits recomputed from the FP8 logits, every operand of both
contractions E4M3-quantised: P with 1x128 blocks along V for dh, P^T, W^T and
h^T with 128 x 128 blocks).

Tolerance from the arithmetic.  Both sides quantise their own P (float32 on
the GPU, float64 rounded to float32 in the oracle), so a code may differ where
x / S lies within rounding distance of an E4M3 rounding boundary; the oracle
marks those elements (x / S within 2^-17 of a boundary) and allows one code
step there.  Everything else is float32 accumulation: each output element is
within 2^-8 of the sum of the absolute values of its quantised terms.  Small
shapes compare every element; grpo_8b compares 64 sampled rows of dh and
bounds the column sums of dW.
"""

import numpy as np
import pytest
import torch

from oracle import e4m3 as OE
from oracle import logprobs as OL
from oracle import quantize as OQ
from paper_2609_22870_gb300 import synth
from tests import oracle_strips
from tests.gpu_helpers import POOL_STRIP, _pool, _w_strips, oracle_logprobs_rows, sample_rows

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


def _flip_slack(x, s):
    """One E4M3 step times the scale where x / s lies within 2^-17 of a
    rounding boundary (the code may differ between two nearby values of x),
    else 0.  x, s broadcastable float64 arrays."""
    q = np.asarray(x, np.float64) / np.asarray(s, np.float64)
    d = 2.0 ** -17
    lo = OE.decode(OE.encode((q * (1 - d)).astype(np.float32)))
    hi = OE.decode(OE.encode((q * (1 + d)).astype(np.float32)))
    return np.abs(hi - lo) * np.asarray(s, np.float64)


def _pow2_flip_slack(x, block_rows):
    """Power-of-two scales (the UE8M0 variant): where a block's amax / 448
    lies within 2^-17 of a power of two, the two sides may pick scales a factor
    of two apart and every code of the block may differ; there each element
    may be off by the E4M3 rounding error at both scales (2 max(2^-4 |x|,
    2^-10 S) with S the larger).  Blocks are block_rows x 128 of x (R, C),
    C a multiple of 128; 0 elsewhere."""
    x = np.abs(np.asarray(x, np.float64))
    R, C = x.shape
    out = np.zeros_like(x)
    d = 2.0 ** -17
    for r0 in range(0, R, block_rows):
        for c0 in range(0, C, 128):
            blk = x[r0:r0 + block_rows, c0:c0 + 128]
            t = float(np.float32(np.float32(blk.max()) / np.float32(448.0))) if blk.size else 0.0
            if t == 0.0:
                continue
            lo, hi = np.ceil(np.log2(t * (1 - d))), np.ceil(np.log2(t * (1 + d)))
            if lo != hi:
                out[r0:r0 + block_rows, c0:c0 + 128] = 2 * np.maximum(2.0 ** -4 * blk, 2.0 ** -10 * 2.0 ** hi)
    return out


def _oracle(h, W, y, g, gran, bwd_pow2=False):
    fwd_pow2 = gran == UE
    pow2 = fwd_pow2 or bwd_pow2
    og = OQ.BLOCK if fwd_pow2 else gran
    h32, W32 = h.float().cpu().numpy(), W.float().cpu().numpy()
    hq, hs = OQ.quantize(h32, og, OQ.ACT, pow2=fwd_pow2)
    wq, ws = OQ.quantize(W32, og, OQ.WEIGHT, pow2=fwd_pow2)
    ref = OL.lm_head_backward_fp8(hq, hs, wq, ws, og, y.cpu().numpy(), g.cpu().numpy(), h32, W32, pow2=pow2)
    T, V = ref["P"].shape
    P = ref["P"].astype(np.float64)
    sp = np.repeat(ref["p_scales"], 128, axis=1)[:, :V]
    spt = np.repeat(np.repeat(ref["pt_scales"], 128, axis=0), 128, axis=1)[:V, :T]
    aw, ah = np.abs(ref["Wt_hat"]).T, np.abs(ref["ht_hat"]).T  # (V, H), (T, H)
    slack_p, slack_pt = _flip_slack(P, sp), _flip_slack(P.T, spt)
    if pow2:
        slack_p = slack_p + _pow2_flip_slack(OL._pad_cols(ref["P"]), 1)[:, :V]
        slack_pt = slack_pt + _pow2_flip_slack(OL._pad_cols(ref["P"].T), 128)[:, :T]
    bound_dh = REL * (np.abs(ref["P_hat"]) @ aw) + slack_p @ aw
    bound_dW = REL * (np.abs(ref["Pt_hat"]) @ ah) + slack_pt @ ah
    return ref, bound_dh, bound_dW


UE = 3  # power-of-two block scales on the block-scaled MMA (forward and backward)


@pytest.mark.parametrize("gran,bwd_pow2", [(OQ.TENSOR, False), (OQ.ROWWISE, False), (OQ.BLOCK, False),
                                           (UE, False), (OQ.BLOCK, True), (OQ.ROWWISE, True)])
@pytest.mark.parametrize("T,H,V", [(300, 256, 1000), (129, 384, 1001), (1, 128, 1), (520, 128, 4096)])
def test_backward_small_all_elements(cuda_lib, gran, bwd_pow2, T, H, V):
    """bwd_pow2: the paper-scale forward with the backward's own operands on
    power-of-two scales (FP8RL_BWD_POW2_SCALES); UE implies it."""
    h, W, y, g = _data(T, H, V, T + V)
    out, _ = _forward_backward(cuda_lib, h, W, y, g, gran, pow2_scales=bwd_pow2)
    ref, bh, bw = _oracle(h, W, y, g, gran, bwd_pow2)
    dh = out["dh"].cpu().numpy().astype(np.float64)
    dW = out["dW"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(dh - ref["dh"]) <= bh + 1e-30)
    assert np.all(np.abs(dW - ref["dW"]) <= bw + 1e-30)
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
    # two chunks of 256 tokens accumulated: the 128 x 128 blocks of P^T and h^T
    # are those of the whole batch (chunk edges fall on block edges), so only
    # the summation order differs
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


@pytest.mark.parametrize("gran,bwd_pow2", [(OQ.BLOCK, False), (OQ.TENSOR, False), (UE, False), (OQ.BLOCK, True)])
def test_backward_full_size_grpo8b(cuda_lib, gran, bwd_pow2):
    """grpo_8b (T 16384, H 4096, V 151936): 64 sampled rows of dh against the
    oracle's FP8 backward; dW by bounded column sums.  UE: power-of-two scales
    on every operand, the contractions on the block-scaled MMA; bwd_pow2: the
    same for the backward's operands after a paper-scale forward."""
    api = cuda_lib
    w = synth.WORKLOADS["grpo_8b"]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    g = (torch.randn(w.T, generator=torch.Generator().manual_seed(8)) / w.T).float().cuda()
    out, _ = _forward_backward(api, h, W, y, g, gran, pow2_scales=bwd_pow2)
    dh = out["dh"]
    assert bool(torch.isfinite(dh).all()) and bool(torch.isfinite(out["dW"]).all())
    rows = sample_rows(w.T, 60, 9)
    pow2 = gran == UE or bwd_pow2
    _, lse_r, z_r = oracle_logprobs_rows(h, W, OQ.BLOCK if gran == UE else gran, y, rows, pow2=gran == UE)
    P = OL.dlogits(z_r, y.cpu().numpy()[rows], lse_r, g.cpu().numpy()[rows]).astype(np.float32)
    Pp = OL._pad_cols(P)
    kw = {"pow2": True, "scale_floor": OQ.E8M0_MIN} if pow2 else {}
    pq, ps = OQ.quantize(Pp, OQ.BLOCK, OQ.ACT, **kw)
    p_hat = OQ.dequantize(pq, ps, OQ.BLOCK, OQ.ACT)
    slack = _flip_slack(Pp, np.repeat(ps, 128, axis=1))
    if pow2:
        slack = slack + _pow2_flip_slack(Pp, 1)
    tasks = ((p_hat[:, v0:v0 + wx.shape[0]], slack[:, v0:v0 + wx.shape[0]], wx, pow2)
             for v0, wx in _w_strips(W, POOL_STRIP))
    ref = np.zeros((len(rows), w.H))
    mag = np.zeros_like(ref)
    slk = np.zeros_like(ref)
    for a, b, c in _pool().map(oracle_strips.bwd_dh_strip, tasks):
        ref += a
        mag += b
        slk += c
    got = dh[torch.as_tensor(rows, device="cuda")].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - ref) <= REL * mag + slk + 1e-30)
    # columns of dW: sum_v dW[v][k] = sum_t (sum_v P_hat[t][v]) h_hat[t][k]; each
    # row of P sums to 0 and E4M3 moves each |P| by at most 2^-4 of itself
    # (plus the subnormal floor), sum_v |P[t][v]| <= 2 |g_t|
    col = out["dW"].double().sum(0)
    lim = 2.0 ** -3 * 1.07 * (g.abs().double()[:, None] * h.double().abs()).sum(0)
    assert bool((col.abs() <= lim + 1e-6 * out["dW"].abs().double().sum(0)).all())
