"""Oracle logits of a vocabulary strip, for a process pool (test side only).

Each z[t][v] of the lm_head is its own dot product, so the oracle's logits can
be evaluated one vocabulary strip at a time and the strips placed side by side:
nothing in the definition changes.  This module imports only numpy and the
oracle, so pool workers started with ``spawn`` load quickly and never touch
CUDA.
"""

import numpy as np

from oracle import logprobs as OL
from oracle import quantize as OQ


def fp8_strip(args):
    """z[:, v0:v1] of the FP8 lm_head: the strip of W quantised by the oracle
    (with the whole tensor's scale in per-tensor mode), then the oracle's
    float64 logits against the already quantised token rows."""
    hq, hs_rows, w_strip, gran, w_tensor_scale, pow2 = args
    if gran == OQ.TENSOR:
        wq = OQ._encode_block(w_strip, w_tensor_scale[0])
        ws = w_tensor_scale
    else:
        wq, ws = OQ.quantize(w_strip, gran, OQ.WEIGHT, pow2=pow2)
    return OL.logits(hq, hs_rows, wq, ws, gran)


def bf16_strip(args):
    """z[:, v0:v1] of the BF16 shadow pass: float64 products of the bf16 values."""
    h_rows, w_strip = args
    return OL.bf16_logits(h_rows, w_strip)


def bwd_dh_strip(args):
    """Partial dh of the FP8 backward over one vocabulary strip: the oracle
    quantises the strip of W with 128 x 128 blocks (the blocks of W^T; with
    pow2 the power-of-two scales of the UE8M0 variant, floored at 2^-127),
    and returns (P_hat[:, strip] @ W_hat_strip, |P_hat[:, strip]| @
    |W_hat_strip|, slack[:, strip] @ |W_hat_strip|) in float64."""
    p_hat, slack, w_strip, pow2 = args
    kw = {"pow2": True, "scale_floor": OQ.E8M0_MIN} if pow2 else {}
    wq, ws = OQ.quantize(w_strip, OQ.BLOCK, OQ.WEIGHT, **kw)
    wd = OQ.dequantize(wq, ws, OQ.BLOCK, OQ.WEIGHT)
    aw = np.abs(wd)
    return p_hat @ wd, np.abs(p_hat) @ aw, slack @ aw
