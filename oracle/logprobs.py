"""FP8 token scoring: logits, log-probs, ratios, dLoss/dlogits -- oracle side.

Test infrastructure only (see ``oracle/__init__.py``).

§2.1 defines the token ratio r_t = pi_theta(y_t|h_t) / pi_old(y_t|h_t); in the
full-pipeline FP8 setting of §3 both probabilities come from FP8-quantised
forward passes.  For the lm_head this is

  z[t, v]   = sum_k  X_tilde_h[t, k] * X_tilde_W[v, k]       (dequantised, Eq. 3)
  logp_t    = z[t, y_t] - log sum_v exp(z[t, v])             (temperature 1)
  r_t       = exp(logp_new_t - logp_old_t)

evaluated here in float64 from the dequantised operands (mathematically equal
to the per-block scaled sum sum_kb S_h S_W sum_k q_h q_W).

Readings: temperature 1 (the paper evaluates at temperature 1.0 and states no
training temperature); the lm_head input and weight are both FP8-quantised at
the same granularity.

dLoss/dlogits follows from the chain rule through log-softmax:
  dL/dz[t, v] = g_t * (1{v == y_t} - exp(z[t, v] - lse_t)),  g_t = dL/dlogp_t.

The BF16 shadow pass (§4, Algorithm 1: the reference ratios r_BF16 come from
forward passes in BF16, recomputed every few steps) scores the same tokens
from the unquantised BF16 operands:

  z[t, v]   = sum_k  h[t, k] * W[v, k]                        (bf16 values)

again in float64, followed by the same log-softmax and gather.

Backward through the lm_head (the step after dLoss/dlogits): with P the
dLoss/dlogits above and the FP8 logits z of the forward pass,

  dh[t, :] = sum_v P[t, v] W[v, :]        dW[v, :] = sum_t P[t, v] h[t, :]

Reading: the quantisers pass the gradient straight through (their derivative
is taken as the identity), so the contractions use the bf16 operands h and W
the codes were quantised from.

FP8 backward (the paper trains with FP8 GEMMs in the backward pass too, §3
and the performance appendix; it prints no quantisation for them): the same
two contractions with every operand E4M3-quantised by Eq. 3 before it is
multiplied.  Readings: each contraction runs along its own K axis (V for dh,
T for dW), so each operand is quantised along that axis; the gradient P gets
the activation granularity of the forward pass, 1x128 blocks along K, where
each thread of a tile holds one token's 128 vocabulary entries (P for dh);
its transpose (the A operand of dW, K = T) gets 128 x 128 blocks, as do the
transposed bf16 weight W^T and hidden states h^T (the B operands; the weight
granularity of the forward pass).  P is taken in float32 (the value the
hardware holds) before it is quantised; V and T are padded with zeros to
multiples of 128 along K.

With power-of-two (UE8M0) forward scales the backward keeps that scale format
for its own four operands (the scales of the hardware's block-scaled MMA):
each S is the smallest power of two not below fl32(amax / 448), raised to
2^-127 where it falls below E8M0's range.
"""

import numpy as np

from . import quantize as Q


def logits(h_codes, h_scales, w_codes, w_scales, gran, rows=None):
    """z = X_tilde_h @ X_tilde_W^T in float64 (optionally for a subset of rows)."""
    xh = Q.dequantize(h_codes, h_scales, gran, Q.ACT)
    if rows is not None:
        xh = xh[np.asarray(rows)]
    xw = Q.dequantize(w_codes, w_scales, gran, Q.WEIGHT)
    return xh @ xw.T


def log_softmax_gather(z, targets):
    """(logp, lse): lse_t = log sum_v exp z[t, v]; logp_t = z[t, y_t] - lse_t."""
    z = np.asarray(z, dtype=np.float64)
    y = np.asarray(targets, dtype=np.int64)
    if np.any(y < 0) or np.any(y >= z.shape[1]):
        raise ValueError("target outside [0, V)")
    m = np.max(z, axis=1)
    lse = m + np.log(np.sum(np.exp(z - m[:, None]), axis=1))
    zy = z[np.arange(z.shape[0]), y]
    return zy - lse, lse


def token_logprobs(h_codes, h_scales, w_codes, w_scales, gran, targets, rows=None):
    """Per-token log-prob (and lse) of the target under the FP8 lm_head."""
    z = logits(h_codes, h_scales, w_codes, w_scales, gran, rows)
    y = np.asarray(targets)
    if rows is not None:
        y = y[np.asarray(rows)]
    return log_softmax_gather(z, y)


def bf16_logits(h, W, rows=None):
    """z = h @ W^T in float64 from the bf16-valued operands (the BF16 shadow
    pass of §4; no quantisation)."""
    h = np.asarray(h, dtype=np.float64)
    if rows is not None:
        h = h[np.asarray(rows)]
    return h @ np.asarray(W, dtype=np.float64).T


def bf16_token_logprobs(h, W, targets, rows=None):
    """Per-token (logp, lse) of the target under the BF16 lm_head (§4 reference pass)."""
    z = bf16_logits(h, W, rows)
    y = np.asarray(targets)
    if rows is not None:
        y = y[np.asarray(rows)]
    return log_softmax_gather(z, y)


def importance_ratios(logp_new, logp_old):
    """r_t = exp(logp_new - logp_old) (§2.1), float64."""
    return np.exp(np.asarray(logp_new, np.float64) - np.asarray(logp_old, np.float64))


def dlogits(z, targets, lse, g):
    """dL/dz[t, v] = g_t (1{v == y_t} - exp(z[t, v] - lse_t)), float64."""
    z = np.asarray(z, dtype=np.float64)
    p = np.exp(z - np.asarray(lse, np.float64)[:, None])
    onehot = np.zeros_like(p)
    onehot[np.arange(z.shape[0]), np.asarray(targets, np.int64)] = 1.0
    return np.asarray(g, np.float64)[:, None] * (onehot - p)


def lm_head_backward(h_codes, h_scales, w_codes, w_scales, gran, targets, g, h, W, rows=None):
    """dLoss/dh and dLoss/dW of the FP8-scored log-probs, given g_t = dL/dlogp_t.

    z from ``logits`` (float64, dequantised operands), lse from
    ``log_softmax_gather``, P from ``dlogits``; then the two contractions with
    the bf16 operands in float64.  With ``rows`` only those tokens are scored
    and only dh for them is returned (dW needs every token)."""
    y = np.asarray(targets, np.int64)
    gg = np.asarray(g, np.float64)
    if rows is not None:
        rows = np.asarray(rows, np.int64)
        y, gg = y[rows], gg[rows]
    z = logits(h_codes, h_scales, w_codes, w_scales, gran, rows)
    _, lse = log_softmax_gather(z, y)
    P = dlogits(z, y, lse, gg)
    W64 = np.asarray(W, np.float32).astype(np.float64)
    out = {"P": P, "lse": lse, "dh": P @ W64}
    if rows is None:
        out["dW"] = P.T @ np.asarray(h, np.float32).astype(np.float64)
    return out


def _pad_cols(x, mult=128):
    """x (rows, cols) float32, zero-padded to a multiple of `mult` columns."""
    rows, cols = x.shape
    cp = -(-cols // mult) * mult
    out = np.zeros((rows, cp), np.float32)
    out[:, :cols] = x
    return out


def lm_head_backward_fp8(h_codes, h_scales, w_codes, w_scales, gran, targets, g, h, W, pow2=False):
    """dLoss/dh and dLoss/dW with both contractions on E4M3 operands.

    P (float64 from the FP8 logits) is rounded to float32 and quantised twice:
    P [T][V] with 1x128 blocks along V (A operand of dh = P W), P^T [V][T]
    with 128 x 128 blocks (A operand of dW = P^T h); W^T [H][V] and h^T [H][T]
    are quantised from the bf16 values with 128 x 128 blocks (B operands).
    ``pow2``: the four take power-of-two scales floored at 2^-127 (the
    backward of the UE8M0 variant).  The products of the dequantised operands
    are summed in float64.  Returns the quantised operands too (codes and
    scales in natural shape)."""
    y = np.asarray(targets, np.int64)
    gg = np.asarray(g, np.float64)
    z = logits(h_codes, h_scales, w_codes, w_scales, gran)
    _, lse = log_softmax_gather(z, y)
    P32 = dlogits(z, y, lse, gg).astype(np.float32)
    T, V = P32.shape
    kw = {"pow2": True, "scale_floor": Q.E8M0_MIN} if pow2 else {}
    pq, ps = Q.quantize(_pad_cols(P32), Q.BLOCK, Q.ACT, **kw)              # (T, V') codes, (T, V'/128)
    ptq, pts = Q.quantize(_pad_cols(P32.T), Q.BLOCK, Q.WEIGHT, **kw)       # (V, T'),  (ceil(V/128), T'/128)
    wtq, wts = Q.quantize(_pad_cols(np.asarray(W, np.float32).T), Q.BLOCK, Q.WEIGHT, **kw)   # (H, V')
    htq, hts = Q.quantize(_pad_cols(np.asarray(h, np.float32).T), Q.BLOCK, Q.WEIGHT, **kw)   # (H, T')
    P_hat = Q.dequantize(pq, ps, Q.BLOCK, Q.ACT)
    Pt_hat = Q.dequantize(ptq, pts, Q.BLOCK, Q.WEIGHT)
    Wt_hat = Q.dequantize(wtq, wts, Q.BLOCK, Q.WEIGHT)
    ht_hat = Q.dequantize(htq, hts, Q.BLOCK, Q.WEIGHT)
    return {"P": P32, "lse": lse, "dh": P_hat @ Wt_hat.T, "dW": Pt_hat @ ht_hat.T,
            "P_hat": P_hat[:, :V], "Pt_hat": Pt_hat[:, :T], "Wt_hat": Wt_hat[:, :V], "ht_hat": ht_hat[:, :T],
            "p_codes": pq, "p_scales": ps, "pt_codes": ptq, "pt_scales": pts,
            "wt_codes": wtq, "wt_scales": wts, "ht_codes": htq, "ht_scales": hts}
