"""Helpers shared by the GPU parity tests (test side only).

The oracle always quantises from the bf16 inputs itself; nothing the CUDA path
produced is fed to it.  For the full lm_head (V = 151936) the oracle's logits
are evaluated one vocabulary strip at a time: each z[t][v] is its own dot
product, so splitting the columns changes nothing in the definition.
"""

import numpy as np
import torch

from oracle import logprobs as OL
from oracle import quantize as OQ

STRIP = 8192  # vocabulary rows per strip (a multiple of 128)


def scales_natural(gpu_scales, rows, cols, gran, role):
    """GPU scale layout -> the oracle's natural shape."""
    s = gpu_scales.detach().cpu().numpy()
    if gran == OQ.TENSOR:
        return s[:1]
    if gran == OQ.ROWWISE:
        return s[:rows]
    nkb = cols // 128
    if role == OQ.ACT:
        return s[: rows * nkb].reshape(nkb, rows).T
    return s[: ((rows + 127) // 128) * nkb].reshape(-1, nkb)


def oracle_logprobs_rows(h_bf16, W_bf16, gran, targets, rows):
    """Oracle (logp, lse, z) for the selected rows, quantising h and W itself.

    Per-tensor scales need the amax of the whole tensor; the other
    granularities need only the rows / strips involved.
    """
    rows = np.asarray(rows, dtype=np.int64)
    V, H = W_bf16.shape
    if gran == OQ.TENSOR:
        hq, hs = OQ.quantize(h_bf16.float().cpu().numpy(), gran, OQ.ACT)
        hq, hs_rows = hq[rows], hs
    else:
        hq, hs_rows = OQ.quantize(h_bf16[torch.as_tensor(rows, device=h_bf16.device)].float().cpu().numpy(),
                                  gran, OQ.ACT)
    w_tensor_scale = None
    if gran == OQ.TENSOR:
        amax = np.float32(0)
        for v0 in range(0, V, STRIP):
            amax = max(amax, np.max(np.abs(W_bf16[v0:v0 + STRIP].float().cpu().numpy())))
        w_tensor_scale = OQ.scale_from_amax(np.float32(amax)).reshape(1)
    zs = []
    for v0 in range(0, V, STRIP):
        v1 = min(V, v0 + STRIP)
        wx = W_bf16[v0:v1].float().cpu().numpy()
        if gran == OQ.TENSOR:
            wq = OQ._encode_block(wx, w_tensor_scale[0])
            ws = w_tensor_scale
        else:
            wq, ws = OQ.quantize(wx, gran, OQ.WEIGHT)
        zs.append(OL.logits(hq, hs_rows, wq, ws, gran))
    z = np.concatenate(zs, axis=1)
    y = np.asarray(targets.cpu().numpy() if torch.is_tensor(targets) else targets)[rows]
    logp, lse = OL.log_softmax_gather(z, y)
    return logp, lse, z


def sample_rows(T, n, seed):
    rng = np.random.default_rng(seed)
    pick = set(rng.choice(T, size=min(n, T), replace=False).tolist())
    pick.update([0, T - 1, min(T - 1, 127), min(T - 1, 128)])
    return np.array(sorted(pick), dtype=np.int64)
