"""Helpers shared by the GPU parity tests (test side only).

The oracle always quantises from the bf16 inputs itself; nothing the CUDA path
produced is fed to it.  For the full lm_head (V = 151936) the oracle's logits
are evaluated one vocabulary strip at a time: each z[t][v] is its own dot
product, so splitting the columns changes nothing in the definition.  Large
cases farm the strips out to a pool of worker processes started with
``spawn`` (a forked child of a process that has used CUDA may hang); the
workers import numpy and the oracle only (``tests/oracle_strips.py``).
"""

import atexit
import concurrent.futures
import multiprocessing
import os

import numpy as np
import torch

from oracle import logprobs as OL
from oracle import quantize as OQ
from tests import oracle_strips

STRIP = 8192       # vocabulary rows per strip (a multiple of 128)
POOL_STRIP = 4096  # strip height handed to one pool task
_POOL = None


def _pool():
    """The process pool of the oracle strips (spawned once per test process,
    one BLAS thread per worker)."""
    global _POOL
    if _POOL is None:
        n = max(1, min(16, os.cpu_count() or 1))
        saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
        for k in saved:
            os.environ[k] = "1"
        try:
            _POOL = concurrent.futures.ProcessPoolExecutor(max_workers=n,
                                                           mp_context=multiprocessing.get_context("spawn"))
            # start every worker now, while the thread limits are in the environment
            list(_POOL.map(abs, range(n)))
        finally:
            for k, v in saved.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v
        atexit.register(_POOL.shutdown)
    return _POOL


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


def _w_strips(W_bf16, step):
    """Host float32 copies of the vocabulary strips of W (bf16 -> float32 is exact)."""
    Wc = W_bf16.detach().cpu()
    for v0 in range(0, Wc.shape[0], step):
        yield v0, Wc[v0:v0 + step].float().numpy()


def _assemble(results, n_rows, V, step):
    z = np.empty((n_rows, V), dtype=np.float64)
    for i, zs in enumerate(results):
        z[:, i * step: i * step + zs.shape[1]] = zs
    return z


def oracle_logits_rows(h_bf16, W_bf16, gran, rows, pow2=False):
    """Oracle FP8 logits z[rows][V] (float64), quantising h and W itself.

    Per-tensor scales need the amax of the whole tensor; the other
    granularities need only the rows / strips involved.
    """
    rows = np.asarray(rows, dtype=np.int64)
    V, H = W_bf16.shape
    if gran == OQ.TENSOR:
        hq, hs = OQ.quantize(h_bf16.float().cpu().numpy(), gran, OQ.ACT, pow2=pow2)
        hq, hs_rows = hq[rows], hs
    else:
        hq, hs_rows = OQ.quantize(h_bf16[torch.as_tensor(rows, device=h_bf16.device)].float().cpu().numpy(),
                                  gran, OQ.ACT, pow2=pow2)
    w_tensor_scale = None
    if gran == OQ.TENSOR:
        amax = np.float32(0)
        for _, wx in _w_strips(W_bf16, STRIP):
            amax = max(amax, np.max(np.abs(wx)))
        f = OQ.pow2_scale_from_amax if pow2 else OQ.scale_from_amax
        w_tensor_scale = np.asarray(f(np.float32(amax)), np.float32).reshape(1)
    big = V * len(rows) * H > (1 << 34)
    if not big:
        zs = [oracle_strips.fp8_strip((hq, hs_rows, wx, gran, w_tensor_scale, pow2))
              for _, wx in _w_strips(W_bf16, STRIP)]
        return np.concatenate(zs, axis=1)
    tasks = ((hq, hs_rows, wx, gran, w_tensor_scale, pow2) for _, wx in _w_strips(W_bf16, POOL_STRIP))
    return _assemble(_pool().map(oracle_strips.fp8_strip, tasks), len(rows), V, POOL_STRIP)


def oracle_logprobs_rows(h_bf16, W_bf16, gran, targets, rows, pow2=False):
    """Oracle (logp, lse, z) for the selected rows (see oracle_logits_rows)."""
    rows = np.asarray(rows, dtype=np.int64)
    z = oracle_logits_rows(h_bf16, W_bf16, gran, rows, pow2=pow2)
    y = np.asarray(targets.cpu().numpy() if torch.is_tensor(targets) else targets)[rows]
    logp, lse = OL.log_softmax_gather(z, y)
    return logp, lse, z


def oracle_bf16_logprobs_rows(h_bf16, W_bf16, targets, rows):
    """Oracle (logp, lse) of the BF16 shadow pass for the selected rows."""
    rows = np.asarray(rows, dtype=np.int64)
    V, H = W_bf16.shape
    hx = h_bf16[torch.as_tensor(rows, device=h_bf16.device)].float().cpu().numpy()
    if V * len(rows) * H > (1 << 34):
        tasks = ((hx, wx) for _, wx in _w_strips(W_bf16, POOL_STRIP))
        z = _assemble(_pool().map(oracle_strips.bf16_strip, tasks), len(rows), V, POOL_STRIP)
    else:
        z = np.concatenate([oracle_strips.bf16_strip((hx, wx)) for _, wx in _w_strips(W_bf16, STRIP)], axis=1)
    y = np.asarray(targets.cpu().numpy() if torch.is_tensor(targets) else targets)[rows]
    return OL.log_softmax_gather(z, y)


def sample_rows(T, n, seed):
    rng = np.random.default_rng(seed)
    pick = set(rng.choice(T, size=min(n, T), replace=False).tolist())
    pick.update([0, T - 1, min(T - 1, 127), min(T - 1, 128)])
    return np.array(sorted(pick), dtype=np.int64)


def full_size_rows(T, seed, n_random=1024, tile=128, band=64 * 128):
    """Rows checked at full size: ``n_random`` random rows, both sides of every
    128-row tile boundary, both sides of every band boundary of the GEMM's
    tile order (64 token tiles), and the first and last rows."""
    rng = np.random.default_rng(seed)
    pick = set(rng.choice(T, size=min(n_random, T), replace=False).tolist())
    for b in range(tile, T, tile):
        pick.update([b - 1, b])
    for b in range(band, T, band):
        pick.update([b - 1, b])
    pick.update([0, T - 1])
    return np.array(sorted(pick), dtype=np.int64)
