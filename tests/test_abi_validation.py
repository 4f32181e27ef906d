"""Host-side argument checks of the C ABI (no GPU needed: every call below is
rejected before any CUDA call, so only the host logic runs)."""

import ctypes
import importlib.util
import os
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def api():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no CUDA toolkit")
    from paper_2609_22870_gb300 import _build
    _build.build()
    spec = importlib.util.spec_from_file_location("_api_validation", os.path.join(
        ROOT, "paper_2609_22870_gb300", "api.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)  # loads the library; calls nothing on the GPU
    return mod


P = ctypes.c_void_p(4096)      # a non-null, 16-byte aligned stand-in (never dereferenced)
ODD = ctypes.c_void_p(4096 + 8)
NULL = None


def _bwd(api, T=64, H=128, V=256, gran=2, h=P, dh=P, dW=P, ws=P, ws_bytes=None, hc=P, lse=P, flags=0):
    if ws_bytes is None:
        ws_bytes = api.lib.fp8rl_lm_head_backward_workspace_size(T, H, V)
    return api.lib.fp8rl_lm_head_backward(hc, P, P, P, gran, T, H, V, P, lse, P, h, P, dh, dW, flags, ws,
                                          ws_bytes, NULL)


def test_lm_head_backward_workspace_size(api):
    T, H, V = 16384, 4096, 151936

    def up(x, a):
        return (x + a - 1) // a * a
    vp, tp, hb = up(V, 128), up(T, 128), up(H, 128) // 128
    # E4M3 codes and float scales of P [T][V'], P^T [V][T'], W^T [H][V'], h^T [H][T'],
    # then the E8M0 scale images of the UE8M0 variant's GEMMs (512 bytes per 128
    # rows of A, 1024 per 256 rows of B, for each group of four 128-wide K
    # blocks), one buffer for the largest of the three: recompute (M T, N V,
    # K H), dh (T, H, V'), dW (V, H, T')
    def images(M, N, K):
        return (up(M, 128) // 128 * 512 + up(N, 256) // 256 * 1024) * ((up(K, 128) // 128 + 3) // 4)
    parts = [T * vp, (vp // 128) * T * 4, V * tp, (tp // 128) * V * 4,
             H * vp, hb * (vp // 128) * 4, H * tp, hb * (tp // 128) * 4,
             max(images(T, V, H), images(T, H, vp), images(V, H, tp))]
    want = sum(up(p, 256) for p in parts)
    assert api.lib.fp8rl_lm_head_backward_workspace_size(T, H, V) == want  # 5.72 GB
    assert api.lib.fp8rl_lm_head_backward_workspace_size(0, H, V) == 0
    assert api.lib.fp8rl_lm_head_backward_workspace_size(T, H, -1) == 0


def test_lm_head_backward_rejects_bad_arguments(api):
    assert _bwd(api, hc=NULL) == api.EINVAL
    assert _bwd(api, flags=4) == api.EINVAL  # unknown flag bit
    assert _bwd(api, flags=api.BWD_ACCUMULATE_DW | api.BWD_POW2_SCALES, hc=NULL) == api.EINVAL
    assert _bwd(api, lse=NULL) == api.EINVAL
    assert _bwd(api, dh=NULL, dW=NULL) == api.EINVAL
    assert _bwd(api, gran=7) == api.EINVAL
    assert _bwd(api, T=0) == api.ESHAPE
    assert _bwd(api, H=100) == api.ESHAPE          # not a multiple of 16
    assert _bwd(api, H=192, gran=2) == api.ESHAPE  # block scaling needs H % 128 == 0
    assert _bwd(api, T=(1 << 31) - 255) == api.ESHAPE  # 32-bit GEMM indices
    assert _bwd(api, V=(1 << 31) - 255) == api.ESHAPE
    assert _bwd(api, h=ODD) == api.EALIGN
    assert _bwd(api, dW=ODD) == api.EALIGN
    assert _bwd(api, ws=NULL) == api.EWORKSPACE
    assert _bwd(api, ws_bytes=1024) == api.EWORKSPACE


def test_seq_level_surrogate_rejects_bad_arguments(api):
    f = api.lib.fp8rl_seq_level_clipped_surrogate
    ws = api.lib.fp8rl_seq_level_surrogate_workspace_size(100, 10)
    assert ws > 0 and api.lib.fp8rl_seq_level_surrogate_workspace_size(-1, 10) == 0
    # stats missing; logp missing with tokens; advantages missing with sequences
    assert f(P, P, P, NULL, P, 10, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, NULL, P, ws, NULL) == api.EINVAL
    assert f(NULL, P, P, NULL, P, 10, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws, NULL) == api.EINVAL
    assert f(P, P, NULL, NULL, P, 10, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws, NULL) == api.EINVAL
    assert f(P, P, P, NULL, P, -1, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws, NULL) == api.ESHAPE
    assert f(P, P, P, NULL, P, 1 << 31, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws, NULL) == api.ESHAPE
    assert f(P, P, P, NULL, P, 10, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws - 1, NULL) \
        == api.EWORKSPACE


def test_seq_mean_surrogate_rejects_bad_arguments(api):
    f = api.lib.fp8rl_clipped_surrogate_seq_mean
    ws = api.lib.fp8rl_surrogate_seq_mean_workspace_size(100, 10)
    assert f(P, P, NULL, NULL, P, 10, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, ws, NULL) == api.EINVAL
    assert f(P, P, NULL, NULL, NULL, 10, 100, 0.8, 1.2, NULL, NULL, NULL, P, P, ws, NULL) == api.EINVAL
    assert f(P, P, NULL, NULL, P, 10, -5, 0.8, 1.2, NULL, NULL, NULL, P, P, ws, NULL) == api.ESHAPE
    assert f(P, P, NULL, NULL, P, 10, 100, 0.8, 1.2, NULL, NULL, NULL, P, NULL, ws, NULL) == api.EWORKSPACE


def test_token_mean_surrogate_rejects_bad_arguments(api):
    # (r, adv, mask, w, T, lo, hi, bounds, n_valid, grad, clip_mask, stats, ws, ws_bytes, stream):
    # the binding's signature table must match the header's, argument for argument
    f = api.lib.fp8rl_clipped_surrogate
    ws = api.lib.fp8rl_surrogate_workspace_size(100)
    assert f(P, P, NULL, NULL, 100, 0.8, 1.2, NULL, P, NULL, NULL, NULL, P, ws, NULL) == api.EINVAL
    assert f(NULL, P, NULL, NULL, 100, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws, NULL) == api.EINVAL
    assert f(P, P, NULL, NULL, -1, 0.8, 1.2, NULL, NULL, NULL, NULL, P, P, ws, NULL) == api.ESHAPE
    assert f(P, P, NULL, NULL, 100, 0.8, 1.2, NULL, P, NULL, NULL, P, NULL, ws, NULL) == api.EWORKSPACE


def test_quantize_ue8m0_rejects_bad_arguments(api):
    f = api.lib.fp8rl_quantize_ue8m0
    assert f(NULL, 4, 128, 128, 2, 0, P, P, NULL, 0, NULL) == api.EINVAL      # no input
    assert f(P, 4, 128, 128, 9, 0, P, P, NULL, 0, NULL) == api.EINVAL         # unknown granularity
    assert f(P, 4, 128, 128, 2, 5, P, P, NULL, 0, NULL) == api.EINVAL         # unknown role
    assert f(P, 4, 192, 192, 2, 0, P, P, NULL, 0, NULL) == api.ESHAPE         # block needs cols % 128
    assert f(P, 4, 128, 100, 1, 0, P, P, NULL, 0, NULL) == api.ESHAPE         # ld < cols
    assert f(ODD, 4, 128, 128, 1, 0, P, P, NULL, 0, NULL) == api.EALIGN
    assert f(P, 4, 128, 128, 0, 0, P, P, NULL, 0, NULL) == api.EWORKSPACE     # per-tensor needs the amax word
