"""Thin Python binding of libfp8rl.so (the C ABI in include/fp8rl.h).

Argument marshalling only: every function here checks tensor placement and
dtypes, allocates outputs and workspaces through torch, and calls the C entry
point of the same name on the current CUDA stream.  All arithmetic happens in
the library's CUDA kernels.  Importing this module loads the library and fails
loudly if it has not been built (``__graft_entry__.build()``).
"""

import ctypes
import math
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libfp8rl.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"libfp8rl.so not built at {_LIB_PATH}; run __graft_entry__.build() first")
lib = ctypes.CDLL(_LIB_PATH)

OK, EINVAL, ESHAPE, EALIGN, EWORKSPACE, ECUDA, EDEVICE, ETIMEOUT = range(8)
GRAN_TENSOR, GRAN_ROWWISE, GRAN_BLOCK = 0, 1, 2
# block layout with power-of-two scales, applied by the block-scaled MMA (scoring calls only)
GRAN_BLOCK_UE8M0 = 3
BWD_ACCUMULATE_DW, BWD_POW2_SCALES = 1, 2  # fp8rl_lm_head_backward flags
ROLE_ACT, ROLE_WEIGHT = 0, 1
CALIB_EXACT, CALIB_GRID = 0, 1
CLIP_HI, CLIP_LO = 1, 2


class CalibOpts(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("lo_min", ctypes.c_double), ("lo_max", ctypes.c_double),
                ("hi_min", ctypes.c_double), ("hi_max", ctypes.c_double),
                ("step", ctypes.c_double), ("delta_lo", ctypes.c_double),
                ("delta_hi", ctypes.c_double), ("lo_old", ctypes.c_float),
                ("hi_old", ctypes.c_float)]


class CalibResult(ctypes.Structure):
    _fields_ = [("lo_new", ctypes.c_float), ("hi_new", ctypes.c_float),
                ("lo_star", ctypes.c_float), ("hi_star", ctypes.c_float),
                ("c_lo", ctypes.c_float), ("c_hi", ctypes.c_float),
                ("flags", ctypes.c_int32), ("shift", ctypes.c_int32),
                ("n_neg", ctypes.c_int64), ("n_pos", ctypes.c_int64),
                ("k_bf16", ctypes.c_int64), ("k_fp8", ctypes.c_int64),
                ("sum_pos_bf16", ctypes.c_int64), ("sum_neg_bf16", ctypes.c_int64),
                ("sum_neg_fp8", ctypes.c_int64), ("sum_pos_fp8", ctypes.c_int64),
                ("rho_bf16", ctypes.c_double), ("rho_fp8", ctypes.c_double),
                ("n_valid", ctypes.c_int64)]


class ClipStats(ctypes.Structure):
    _fields_ = [("loss", ctypes.c_double), ("loss_sum", ctypes.c_double),
                ("n_valid", ctypes.c_int64), ("n_pos", ctypes.c_int64), ("n_neg", ctypes.c_int64),
                ("clipped_pos", ctypes.c_int64), ("clipped_neg", ctypes.c_int64),
                ("lo", ctypes.c_float), ("hi", ctypes.c_float),
                ("flags", ctypes.c_int32), ("n_seq_valid", ctypes.c_int32),
                ("clip_frac_pos", ctypes.c_double), ("clip_frac_neg", ctypes.c_double),
                ("clip_frac", ctypes.c_double)]


class ClipDiag(ctypes.Structure):
    _fields_ = [("n_valid", ctypes.c_int64), ("n_pos", ctypes.c_int64), ("n_neg", ctypes.c_int64),
                ("clipped_lo_fp8", ctypes.c_int64), ("clipped_hi_fp8", ctypes.c_int64),
                ("clipped_lo_bf16", ctypes.c_int64), ("clipped_hi_bf16", ctypes.c_int64),
                ("over_clipped_lo", ctypes.c_int64), ("over_clipped_hi", ctypes.c_int64),
                ("abs_err_prob", ctypes.c_double), ("sum_prob_bf16", ctypes.c_double),
                ("abs_err_ratio", ctypes.c_double), ("sum_ratio_bf16", ctypes.c_double),
                ("nmae_prob", ctypes.c_double), ("nmae_ratio", ctypes.c_double),
                ("c_lo", ctypes.c_float), ("c_hi", ctypes.c_float),
                ("flags", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_p, _i64, _u64, _f, _i, _sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_float,
                               ctypes.c_int, ctypes.c_size_t)
_SIGS = {
    "fp8rl_check": (_i, [_p]),
    "fp8rl_status_string": (ctypes.c_char_p, [_i]),
    "fp8rl_last_cuda_error": (ctypes.c_char_p, []),
    "fp8rl_scales_count": (_i64, [_i64, _i64, _i, _i]),
    "fp8rl_quantize_workspace_size": (_sz, [_i64, _i64, _i, _i]),
    "fp8rl_quantize": (_i, [_p, _i64, _i64, _i64, _i, _i, _p, _p, _p, _sz, _p]),
    "fp8rl_quantize_ue8m0": (_i, [_p, _i64, _i64, _i64, _i, _i, _p, _p, _p, _sz, _p]),
    "fp8rl_token_logprobs_workspace_size": (_sz, [_i64, _i64, _i64, _i]),
    "fp8rl_token_logprobs": (_i, [_p, _p, _p, _p, _i, _i64, _i64, _i64, _p, _p, _p, _p, _p, _p, _sz, _p]),
    "fp8rl_logit_partials": (_i, [_p, _p, _p, _p, _i, _i64, _i64, _i64, _p, _p, _sz, _p]),
    "fp8rl_combine_logprobs": (_i, [_i64, _i64, _i64, _i, _p, _p, _p, _p, _p, _p, _sz, _p]),
    "fp8rl_importance_ratios": (_i, [_p, _p, _i64, _p, _p]),
    "fp8rl_bf16_token_logprobs_workspace_size": (_sz, [_i64, _i64, _i64]),
    "fp8rl_bf16_token_logprobs": (_i, [_p, _i64, _p, _i64, _i64, _i64, _i64, _p, _p, _p, _p, _p, _p,
                                       _sz, _p]),
    "fp8rl_token_logprobs_noalloc": (_i, [_p, _p, _p, _p, _i, _i64, _i64, _i64, _p, _p, _p, _p, _p, _p]),
    "fp8rl_default_calib_opts": (None, [ctypes.POINTER(CalibOpts)]),
    "fp8rl_calibrate_workspace_size": (_sz, [_i64]),
    "fp8rl_calibrate_clip_bounds": (_i, [_p, _p, _p, _p, _p, _i64, _f, _f, ctypes.POINTER(CalibOpts),
                                         _p, _p, _sz, _p]),
    "fp8rl_surrogate_workspace_size": (_sz, [_i64]),
    "fp8rl_clipped_surrogate": (_i, [_p, _p, _p, _p, _i64, _f, _f, _p, _p, _p, _p, _p, _p, _sz, _p]),
    "fp8rl_dlogits_workspace_size": (_sz, [_i64, _i64, _i64, _i]),
    "fp8rl_dlogits_rows": (_i, [_p, _p, _p, _p, _i, _i64, _i64, _i64, _p, _p, _p, _p, _i64, _p, _p,
                                _sz, _p]),
    "fp8rl_surrogate_seq_mean_workspace_size": (_sz, [_i64, _i64]),
    "fp8rl_clipped_surrogate_seq_mean": (_i, [_p, _p, _p, _p, _p, _i64, _i64, _f, _f, _p, _p, _p, _p, _p,
                                              _sz, _p]),
    "fp8rl_lm_head_backward_workspace_size": (_sz, [_i64, _i64, _i64]),
    "fp8rl_lm_head_backward": (_i, [_p, _p, _p, _p, _i, _i64, _i64, _i64, _p, _p, _p, _p, _p, _p, _p, _i,
                                    _p, _sz, _p]),
    "fp8rl_seq_level_surrogate_workspace_size": (_sz, [_i64, _i64]),
    "fp8rl_seq_level_clipped_surrogate": (_i, [_p, _p, _p, _p, _p, _i64, _i64, _f, _f, _p, _p, _p, _p, _p,
                                               _p, _sz, _p]),
    "fp8rl_clip_diagnostics_workspace_size": (_sz, [_i64]),
    "fp8rl_clip_diagnostics": (_i, [_p, _p, _p, _p, _p, _p, _i64, _f, _f, _p, _p, _sz, _p]),
    "fp8rl_tis_weights": (_i, [_p, _p, _i64, _f, _p, _p]),
    "fp8rl_set_wait_limit_ns": (None, [_u64]),
    "fp8rl_wait_selftest": (_i, [_u64, _p]),
}
for _name, (_res, _args) in _SIGS.items():
    _fn = getattr(lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args


class Fp8rlError(RuntimeError):
    def __init__(self, status, where):
        msg = lib.fp8rl_status_string(status).decode()
        if status == ECUDA:
            msg += ": " + lib.fp8rl_last_cuda_error().decode()
        super().__init__(f"{where}: {msg} (status {status})")
        self.status = status


def _ok(status, where):
    if status != OK:
        raise Fp8rlError(status, where)


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dev(t, dtype, name, numel=None):
    if t is None:
        return None
    if not t.is_cuda or t.dtype != dtype or not t.is_contiguous():
        raise ValueError(f"{name}: expected a contiguous CUDA {dtype} tensor")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name}: expected {numel} elements, got {t.numel()}")
    return t


def _workspace(nbytes, device):
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


def check(stream=None):
    """fp8rl_check: synchronise and raise on a device-flagged error."""
    _ok(lib.fp8rl_check(_stream(stream)), "fp8rl_check")


def check_status(stream=None):
    """fp8rl_check, returning the status code instead of raising."""
    return lib.fp8rl_check(_stream(stream))


def set_wait_limit_ns(ns):
    lib.fp8rl_set_wait_limit_ns(int(ns))


def wait_selftest(limit_ns, stream=None):
    _ok(lib.fp8rl_wait_selftest(int(limit_ns), _stream(stream)), "fp8rl_wait_selftest")


# ------------------------------------------------------------------ quantize
def scales_count(rows, cols, gran, role):
    return int(lib.fp8rl_scales_count(rows, cols, gran, role))


def quantize(x, gran, role=ROLE_ACT, codes=None, scales=None, workspace=None, stream=None, ue8m0=False):
    """fp8rl_quantize of a 2-D bf16 CUDA tensor -> (codes uint8, scales float32);
    with ``ue8m0`` fp8rl_quantize_ue8m0 (power-of-two scales)."""
    if x.dim() != 2 or x.dtype != torch.bfloat16 or not x.is_cuda or x.stride(1) != 1:
        raise ValueError("x: expected a 2-D CUDA bf16 tensor with unit column stride")
    if gran == GRAN_BLOCK_UE8M0:  # the block layout with power-of-two scales
        gran, ue8m0 = GRAN_BLOCK, True
    rows, cols = x.shape
    n = scales_count(rows, cols, gran, role)
    codes = torch.empty(rows, cols, dtype=torch.uint8, device=x.device) if codes is None else codes
    scales = torch.empty(max(n, 1), dtype=torch.float32, device=x.device) if scales is None else scales
    _dev(codes, torch.uint8, "codes", rows * cols)
    _dev(scales, torch.float32, "scales")
    if scales.numel() < n:
        raise ValueError(f"scales: expected at least {n} elements, got {scales.numel()}")
    wsz = lib.fp8rl_quantize_workspace_size(rows, cols, gran, role)
    if workspace is None and wsz:
        workspace = _workspace(wsz, x.device)
    fn = lib.fp8rl_quantize_ue8m0 if ue8m0 else lib.fp8rl_quantize
    _ok(fn(_ptr(x), rows, cols, x.stride(0), gran, role, _ptr(codes), _ptr(scales),
           _ptr(workspace), 0 if workspace is None else workspace.numel(),
           _stream(stream)), "fp8rl_quantize_ue8m0" if ue8m0 else "fp8rl_quantize")
    return codes, scales


# ------------------------------------------------------------------ scoring
def token_logprobs_workspace_size(T, H, V, gran):
    return int(lib.fp8rl_token_logprobs_workspace_size(T, H, V, gran))


def _gemm_args(h_codes, h_scales, w_codes, w_scales, targets, gran):
    T, H = h_codes.shape
    V = w_codes.shape[0]
    _dev(h_codes, torch.uint8, "h_codes")
    _dev(w_codes, torch.uint8, "w_codes")
    _dev(h_scales, torch.float32, "h_scales")
    _dev(w_scales, torch.float32, "w_scales")
    _dev(targets, torch.int32, "targets", T)
    if w_codes.shape[1] != H:
        raise ValueError("h_codes and w_codes disagree on the hidden size")
    if h_scales.numel() < scales_count(T, H, gran, ROLE_ACT) or \
            w_scales.numel() < scales_count(V, H, gran, ROLE_WEIGHT):
        raise ValueError("h_scales / w_scales: fewer scales than the granularity needs")
    return T, H, V


def token_logprobs(h_codes, h_scales, w_codes, w_scales, gran, targets, logp_old=None,
                   want_lse=True, want_ratio=None, workspace=None, out=None, stream=None):
    """fp8rl_token_logprobs -> dict(logp, lse, ratio) of float32 [T] tensors."""
    T, H, V = _gemm_args(h_codes, h_scales, w_codes, w_scales, targets, gran)
    dev = h_codes.device
    want_ratio = logp_old is not None if want_ratio is None else want_ratio
    _dev(logp_old, torch.float32, "logp_old", T)
    o = out or {}
    logp = o.get("logp", torch.empty(T, dtype=torch.float32, device=dev))
    lse = o.get("lse", torch.empty(T, dtype=torch.float32, device=dev)) if want_lse else None
    ratio = o.get("ratio", torch.empty(T, dtype=torch.float32, device=dev)) if want_ratio else None
    if workspace is None:
        workspace = _workspace(token_logprobs_workspace_size(T, H, V, gran), dev)
    _ok(lib.fp8rl_token_logprobs(_ptr(h_codes), _ptr(h_scales), _ptr(w_codes), _ptr(w_scales), gran,
                                 T, H, V, _ptr(targets), _ptr(logp_old), _ptr(logp), _ptr(lse),
                                 _ptr(ratio), _ptr(workspace), workspace.numel(), _stream(stream)),
        "fp8rl_token_logprobs")
    return {"logp": logp, "lse": lse, "ratio": ratio}


def token_logprobs_noalloc(h_codes, h_scales, w_codes, w_scales, gran, targets, logp_old=None,
                           want_lse=True, want_ratio=None, out=None, stream=None):
    """fp8rl_token_logprobs_noalloc: like token_logprobs, but the scratch is the
    library's fixed static array, for callers that cannot allocate a workspace
    (shapes needing more than FP8RL_NOALLOC_SCRATCH_BYTES are refused)."""
    T, H, V = _gemm_args(h_codes, h_scales, w_codes, w_scales, targets, gran)
    dev = h_codes.device
    want_ratio = logp_old is not None if want_ratio is None else want_ratio
    _dev(logp_old, torch.float32, "logp_old", T)
    o = out or {}
    logp = o.get("logp", torch.empty(T, dtype=torch.float32, device=dev))
    lse = o.get("lse", torch.empty(T, dtype=torch.float32, device=dev)) if want_lse else None
    ratio = o.get("ratio", torch.empty(T, dtype=torch.float32, device=dev)) if want_ratio else None
    _ok(lib.fp8rl_token_logprobs_noalloc(_ptr(h_codes), _ptr(h_scales), _ptr(w_codes), _ptr(w_scales),
                                         gran, T, H, V, _ptr(targets), _ptr(logp_old), _ptr(logp),
                                         _ptr(lse), _ptr(ratio), _stream(stream)),
        "fp8rl_token_logprobs_noalloc")
    return {"logp": logp, "lse": lse, "ratio": ratio}


def logit_partials(h_codes, h_scales, w_codes, w_scales, gran, targets, workspace, stream=None):
    """fp8rl_logit_partials: the FP8 GEMM + streaming logsumexp half."""
    T, H, V = _gemm_args(h_codes, h_scales, w_codes, w_scales, targets, gran)
    _ok(lib.fp8rl_logit_partials(_ptr(h_codes), _ptr(h_scales), _ptr(w_codes), _ptr(w_scales), gran,
                                 T, H, V, _ptr(targets), _ptr(workspace), workspace.numel(),
                                 _stream(stream)), "fp8rl_logit_partials")


def combine_logprobs(T, H, V, gran, targets, workspace, logp_old=None, logp=None, lse=None,
                     ratio=None, stream=None):
    """fp8rl_combine_logprobs: merge the partials left by logit_partials."""
    _ok(lib.fp8rl_combine_logprobs(T, H, V, gran, _ptr(targets), _ptr(logp_old), _ptr(logp),
                                   _ptr(lse), _ptr(ratio), _ptr(workspace), workspace.numel(),
                                   _stream(stream)), "fp8rl_combine_logprobs")


def bf16_token_logprobs_workspace_size(T, H, V):
    return int(lib.fp8rl_bf16_token_logprobs_workspace_size(T, H, V))


def bf16_token_logprobs(h, W, targets, logp_old=None, want_lse=True, want_ratio=None,
                        workspace=None, out=None, stream=None):
    """fp8rl_bf16_token_logprobs: the BF16 shadow pass (unquantised bf16 h, W)
    -> dict(logp, lse, ratio) of float32 [T] tensors."""
    for name, x in (("h", h), ("W", W)):
        if x.dim() != 2 or x.dtype != torch.bfloat16 or not x.is_cuda or x.stride(1) != 1:
            raise ValueError(f"{name}: expected a 2-D CUDA bf16 tensor with unit column stride")
    T, H = h.shape
    V = W.shape[0]
    if W.shape[1] != H:
        raise ValueError("h and W disagree on the hidden size")
    _dev(targets, torch.int32, "targets", T)
    _dev(logp_old, torch.float32, "logp_old", T)
    dev = h.device
    want_ratio = logp_old is not None if want_ratio is None else want_ratio
    o = out or {}
    logp = o.get("logp", torch.empty(T, dtype=torch.float32, device=dev))
    lse = o.get("lse", torch.empty(T, dtype=torch.float32, device=dev)) if want_lse else None
    ratio = o.get("ratio", torch.empty(T, dtype=torch.float32, device=dev)) if want_ratio else None
    if workspace is None:
        workspace = _workspace(bf16_token_logprobs_workspace_size(T, H, V), dev)
    _ok(lib.fp8rl_bf16_token_logprobs(_ptr(h), h.stride(0), _ptr(W), W.stride(0), T, H, V,
                                      _ptr(targets), _ptr(logp_old), _ptr(logp), _ptr(lse),
                                      _ptr(ratio), _ptr(workspace), workspace.numel(),
                                      _stream(stream)), "fp8rl_bf16_token_logprobs")
    return {"logp": logp, "lse": lse, "ratio": ratio}


def importance_ratios(logp_new, logp_old, out=None, stream=None):
    T = logp_new.numel()
    _dev(logp_new, torch.float32, "logp_new")
    _dev(logp_old, torch.float32, "logp_old", T)
    out = torch.empty_like(logp_new) if out is None else out
    _ok(lib.fp8rl_importance_ratios(_ptr(logp_new), _ptr(logp_old), T, _ptr(out), _stream(stream)),
        "fp8rl_importance_ratios")
    return out


# ------------------------------------------------------------------ calibrate
def default_calib_opts():
    o = CalibOpts()
    lib.fp8rl_default_calib_opts(ctypes.byref(o))
    return o


def calib_opts(**kw):
    o = default_calib_opts()
    for k, v in kw.items():
        setattr(o, k, v)
    return o


def calibrate_workspace_size(T):
    return int(lib.fp8rl_calibrate_workspace_size(T))


def calibrate_clip_bounds(r_fp8, r_bf16, adv, mask, coef, eps_low, eps_high, opts=None,
                          result=None, workspace=None, stream=None):
    """fp8rl_calibrate_clip_bounds -> device uint8 buffer holding a CalibResult.

    ``read_calib_result(buf)`` decodes it on the host (synchronising);
    ``bounds_view(buf)`` is the float32 [2] view {lo_new, hi_new} on the device.
    """
    T = r_fp8.numel()
    dev = r_fp8.device
    for t, n, dt in ((r_fp8, "r_fp8", torch.float32), (r_bf16, "r_bf16", torch.float32),
                     (adv, "adv", torch.float32)):
        _dev(t, dt, n, T)
    _dev(mask, torch.uint8, "mask", T)
    _dev(coef, torch.float32, "coef", T)
    result = torch.zeros(ctypes.sizeof(CalibResult), dtype=torch.uint8, device=dev) if result is None else result
    if workspace is None:
        workspace = _workspace(calibrate_workspace_size(T), dev)
    o = default_calib_opts() if opts is None else opts
    _ok(lib.fp8rl_calibrate_clip_bounds(_ptr(r_fp8), _ptr(r_bf16), _ptr(adv), _ptr(mask), _ptr(coef), T,
                                        eps_low, eps_high, ctypes.byref(o), _ptr(result),
                                        _ptr(workspace), workspace.numel(), _stream(stream)),
        "fp8rl_calibrate_clip_bounds")
    return result


def read_calib_result(buf):
    raw = bytes(buf.cpu().numpy().tobytes())
    r = CalibResult.from_buffer_copy(raw)
    return {f: getattr(r, f) for f, _ in CalibResult._fields_}


def bounds_view(buf):
    return buf[:8].view(torch.float32)


def n_valid_view(buf):
    """The valid-token count inside a device fp8rl_calib_result buffer (int64
    [1]), for clipped_surrogate(n_valid=...)."""
    off = CalibResult.n_valid.offset
    return buf[off:off + 8].view(torch.int64)


# ------------------------------------------------------------------ surrogate
def surrogate_workspace_size(T):
    return int(lib.fp8rl_surrogate_workspace_size(T))


def clipped_surrogate(r, adv, mask=None, w_tis=None, lo=0.8, hi=1.2, bounds=None, want_grad=True,
                      want_clip_mask=True, stats=None, workspace=None, out=None, stream=None, n_valid=None):
    """fp8rl_clipped_surrogate -> dict(stats=<device buffer>, grad, clip_mask).
    ``n_valid``: device int64 [1] count of the mask's valid tokens when known
    (n_valid_view of the calibration's result on the same mask), else counted."""
    T = r.numel()
    dev = r.device
    _dev(r, torch.float32, "r")
    _dev(adv, torch.float32, "adv", T)
    _dev(mask, torch.uint8, "mask", T)
    _dev(w_tis, torch.float32, "w_tis", T)
    _dev(bounds, torch.float32, "bounds", 2)
    _dev(n_valid, torch.int64, "n_valid", 1)
    o = out or {}
    grad = o.get("grad", torch.empty(T, dtype=torch.float32, device=dev)) if want_grad else None
    cm = o.get("clip_mask", torch.empty(T, dtype=torch.uint8, device=dev)) if want_clip_mask else None
    stats = torch.zeros(ctypes.sizeof(ClipStats), dtype=torch.uint8, device=dev) if stats is None else stats
    if workspace is None:
        workspace = _workspace(surrogate_workspace_size(T), dev)
    _ok(lib.fp8rl_clipped_surrogate(_ptr(r), _ptr(adv), _ptr(mask), _ptr(w_tis), T, lo, hi,
                                    _ptr(bounds), _ptr(n_valid), _ptr(grad), _ptr(cm), _ptr(stats),
                                    _ptr(workspace), workspace.numel(), _stream(stream)),
        "fp8rl_clipped_surrogate")
    return {"stats": stats, "grad": grad, "clip_mask": cm}


def clipped_surrogate_seq_mean(r, adv, seq_id, n_seq, mask=None, w_tis=None, lo=0.8, hi=1.2, bounds=None,
                               want_grad=True, want_clip_mask=True, stats=None, workspace=None, out=None,
                               stream=None):
    """fp8rl_clipped_surrogate_seq_mean (GRPO per-response normalisation)
    -> dict(stats=<device buffer>, grad, clip_mask)."""
    T = r.numel()
    dev = r.device
    _dev(r, torch.float32, "r")
    _dev(adv, torch.float32, "adv", T)
    _dev(seq_id, torch.int32, "seq_id", T)
    _dev(mask, torch.uint8, "mask", T)
    _dev(w_tis, torch.float32, "w_tis", T)
    _dev(bounds, torch.float32, "bounds", 2)
    o = out or {}
    grad = o.get("grad", torch.empty(T, dtype=torch.float32, device=dev)) if want_grad else None
    cm = o.get("clip_mask", torch.empty(T, dtype=torch.uint8, device=dev)) if want_clip_mask else None
    stats = torch.zeros(ctypes.sizeof(ClipStats), dtype=torch.uint8, device=dev) if stats is None else stats
    if workspace is None:
        workspace = _workspace(lib.fp8rl_surrogate_seq_mean_workspace_size(T, n_seq), dev)
    _ok(lib.fp8rl_clipped_surrogate_seq_mean(_ptr(r), _ptr(adv), _ptr(mask), _ptr(w_tis), _ptr(seq_id),
                                             n_seq, T, lo, hi, _ptr(bounds), _ptr(grad), _ptr(cm),
                                             _ptr(stats), _ptr(workspace), workspace.numel(),
                                             _stream(stream)), "fp8rl_clipped_surrogate_seq_mean")
    return {"stats": stats, "grad": grad, "clip_mask": cm}


def seq_level_clipped_surrogate(logp, logp_old, adv_seq, seq_id, mask=None, lo=0.8, hi=1.2, bounds=None,
                                want_grad=True, stats=None, workspace=None, out=None, stream=None):
    """fp8rl_seq_level_clipped_surrogate (one geometric-mean ratio per
    response, clipped like a token ratio) -> dict(stats=<device buffer>,
    seq_ratio, seq_clip, grad).  ``adv_seq`` holds one advantage per sequence;
    its length is n_seq."""
    T = logp.numel()
    n_seq = adv_seq.numel()
    dev = logp.device
    _dev(logp, torch.float32, "logp")
    _dev(logp_old, torch.float32, "logp_old", T)
    _dev(adv_seq, torch.float32, "adv_seq")
    _dev(seq_id, torch.int32, "seq_id", T)
    _dev(mask, torch.uint8, "mask", T)
    _dev(bounds, torch.float32, "bounds", 2)
    o = out or {}
    ratio = o.get("seq_ratio", torch.empty(n_seq, dtype=torch.float32, device=dev))
    clip = o.get("seq_clip", torch.empty(n_seq, dtype=torch.uint8, device=dev))
    grad = o.get("grad", torch.empty(T, dtype=torch.float32, device=dev)) if want_grad else None
    stats = torch.zeros(ctypes.sizeof(ClipStats), dtype=torch.uint8, device=dev) if stats is None else stats
    if workspace is None:
        workspace = _workspace(lib.fp8rl_seq_level_surrogate_workspace_size(T, n_seq), dev)
    _ok(lib.fp8rl_seq_level_clipped_surrogate(_ptr(logp), _ptr(logp_old), _ptr(adv_seq), _ptr(mask),
                                              _ptr(seq_id), n_seq, T, lo, hi, _ptr(bounds), _ptr(ratio),
                                              _ptr(clip), _ptr(grad), _ptr(stats), _ptr(workspace),
                                              workspace.numel(), _stream(stream)),
        "fp8rl_seq_level_clipped_surrogate")
    return {"stats": stats, "seq_ratio": ratio, "seq_clip": clip, "grad": grad}


def lm_head_backward(h_codes, h_scales, w_codes, w_scales, gran, targets, lse, grad_logp, h, W,
                     want_dh=True, want_dw=True, accumulate_dw=False, pow2_scales=False, out=None,
                     workspace=None, stream=None):
    """fp8rl_lm_head_backward -> dict(dh=[T][H] float32, dW=[V][H] float32).
    ``h`` [T][H] and ``W`` [V][H] are the bf16 operands the codes came from;
    ``out`` may hold preallocated "dh" / "dW" (with ``accumulate_dw`` the
    given dW is added to); ``pow2_scales``: the contractions' operands take
    power-of-two scales on the block-scaled MMA (FP8RL_BWD_POW2_SCALES)."""
    T, H, V = _gemm_args(h_codes, h_scales, w_codes, w_scales, targets, gran)
    dev = h.device
    _dev(lse, torch.float32, "lse", T)
    _dev(grad_logp, torch.float32, "grad_logp", T)
    _dev(h, torch.bfloat16, "h", T * H)
    _dev(W, torch.bfloat16, "W", V * H)
    o = out or {}
    dh = (o.get("dh") if o.get("dh") is not None else torch.empty(T, H, dtype=torch.float32, device=dev)) \
        if want_dh else None
    dW = (o.get("dW") if o.get("dW") is not None else torch.empty(V, H, dtype=torch.float32, device=dev)) \
        if want_dw else None
    _dev(dh, torch.float32, "dh", T * H)
    _dev(dW, torch.float32, "dW", V * H)
    if workspace is None:
        workspace = _workspace(lib.fp8rl_lm_head_backward_workspace_size(T, H, V), dev)
    flags = (BWD_ACCUMULATE_DW if accumulate_dw else 0) | (BWD_POW2_SCALES if pow2_scales else 0)
    _ok(lib.fp8rl_lm_head_backward(_ptr(h_codes), _ptr(h_scales), _ptr(w_codes), _ptr(w_scales), int(gran),
                                   T, H, V, _ptr(targets), _ptr(lse), _ptr(grad_logp), _ptr(h), _ptr(W),
                                   _ptr(dh), _ptr(dW), flags, _ptr(workspace),
                                   workspace.numel(), _stream(stream)), "fp8rl_lm_head_backward")
    return {"dh": dh, "dW": dW}


def read_clip_stats(buf):
    raw = bytes(buf.cpu().numpy().tobytes())
    s = ClipStats.from_buffer_copy(raw)
    return {f: getattr(s, f) for f, _ in ClipStats._fields_}


# ------------------------------------------------------------------ diagnostics
def clip_diagnostics(r_fp8, r_bf16, adv, mask=None, logp_fp8=None, logp_bf16=None, eps_low=0.2,
                     eps_high=0.2, out=None, workspace=None, stream=None):
    """fp8rl_clip_diagnostics (§3): over-clipping, clip counts and NMAE against
    BF16 references -> device buffer holding one fp8rl_clip_diag."""
    T = r_fp8.numel()
    for name, t in (("r_fp8", r_fp8), ("r_bf16", r_bf16), ("adv", adv), ("logp_fp8", logp_fp8),
                    ("logp_bf16", logp_bf16)):
        _dev(t, torch.float32, name, T)
    _dev(mask, torch.uint8, "mask", T)
    dev = r_fp8.device
    out = torch.zeros(ctypes.sizeof(ClipDiag), dtype=torch.uint8, device=dev) if out is None else out
    if workspace is None:
        workspace = _workspace(lib.fp8rl_clip_diagnostics_workspace_size(T), dev)
    _ok(lib.fp8rl_clip_diagnostics(_ptr(logp_fp8), _ptr(logp_bf16), _ptr(r_fp8), _ptr(r_bf16), _ptr(adv),
                                   _ptr(mask), T, eps_low, eps_high, _ptr(out), _ptr(workspace),
                                   workspace.numel(), _stream(stream)), "fp8rl_clip_diagnostics")
    return out


def read_clip_diag(buf):
    raw = bytes(buf.cpu().numpy().tobytes())
    d = ClipDiag.from_buffer_copy(raw[: ctypes.sizeof(ClipDiag)])
    return {name: getattr(d, name) for name, _ in ClipDiag._fields_}


def tis_weights(logp_old, logp_sampler, C=2.0, out=None, stream=None):
    """fp8rl_tis_weights (§2.3): w = min(exp(logp_old - logp_sampler), C)."""
    T = logp_old.numel()
    _dev(logp_old, torch.float32, "logp_old", T)
    _dev(logp_sampler, torch.float32, "logp_sampler", T)
    out = torch.empty(T, dtype=torch.float32, device=logp_old.device) if out is None else out
    _dev(out, torch.float32, "out", T)
    _ok(lib.fp8rl_tis_weights(_ptr(logp_old), _ptr(logp_sampler), T, C, _ptr(out), _stream(stream)),
        "fp8rl_tis_weights")
    return out


# ------------------------------------------------------------------ dlogits
def dlogits_rows(h_codes, h_scales, w_codes, w_scales, gran, targets, lse, grad_logp, rows,
                 out=None, workspace=None, stream=None):
    """fp8rl_dlogits_rows -> float32 [n_rows][V] dense dLoss/dlogits."""
    T, H, V = _gemm_args(h_codes, h_scales, w_codes, w_scales, targets, gran)
    _dev(lse, torch.float32, "lse", T)
    _dev(grad_logp, torch.float32, "grad_logp", T)
    _dev(rows, torch.int64, "rows")
    n = rows.numel()
    dev = h_codes.device
    out = torch.empty(n, V, dtype=torch.float32, device=dev) if out is None else out
    if workspace is None:
        workspace = _workspace(lib.fp8rl_dlogits_workspace_size(n, H, V, gran), dev)
    _ok(lib.fp8rl_dlogits_rows(_ptr(h_codes), _ptr(h_scales), _ptr(w_codes), _ptr(w_scales), gran, T, H,
                               V, _ptr(targets), _ptr(lse), _ptr(grad_logp), _ptr(rows), n, _ptr(out),
                               _ptr(workspace), workspace.numel(), _stream(stream)),
        "fp8rl_dlogits_rows")
    return out


# ------------------------------------------------------------------ whole step
class StepBuffers:
    """Preallocated outputs and workspaces for ``score_calibrate_loss``."""

    def __init__(self, T, H, V, gran, device):
        f32 = dict(dtype=torch.float32, device=device)
        self.h_codes = torch.empty(T, H, dtype=torch.uint8, device=device)
        self.h_scales = torch.empty(max(1, scales_count(T, H, gran, ROLE_ACT)), **f32)
        self.w_codes = torch.empty(V, H, dtype=torch.uint8, device=device)
        self.w_scales = torch.empty(max(1, scales_count(V, H, gran, ROLE_WEIGHT)), **f32)
        self.q_ws = _workspace(max(lib.fp8rl_quantize_workspace_size(T, H, gran, ROLE_ACT),
                                   lib.fp8rl_quantize_workspace_size(V, H, gran, ROLE_WEIGHT), 256), device)
        self.lp_ws = _workspace(token_logprobs_workspace_size(T, H, V, gran), device)
        self.logp = torch.empty(T, **f32)
        self.lse = torch.empty(T, **f32)
        self.ratio = torch.empty(T, **f32)
        self.cal_ws = _workspace(calibrate_workspace_size(T), device)
        self.cal_res = torch.zeros(ctypes.sizeof(CalibResult), dtype=torch.uint8, device=device)
        self.sur_ws = _workspace(surrogate_workspace_size(T), device)
        self.stats = torch.zeros(ctypes.sizeof(ClipStats), dtype=torch.uint8, device=device)
        self.grad = torch.empty(T, **f32)
        self.clip_mask = torch.empty(T, dtype=torch.uint8, device=device)


class HostBatchPrefetcher:
    """Double-buffered host -> device staging of each step's inputs on a side
    stream, so the copy of step i + 1 overlaps the work of step i (the batch
    prefetch of a training loop).  Copies and stream events only.

    ``host`` maps names to pinned CPU tensors; ``prefetch(slot, host)`` copies
    them into device slot ``slot`` (0 or 1) once that slot's previous user has
    released it; ``acquire(slot)`` makes the compute stream wait for the copy
    and returns the slot's device tensors; ``release(slot)`` marks them free
    after the work queued so far on the compute stream."""

    def __init__(self, host, device, stream=None):
        self.device = torch.device(device)
        self.bufs = [{k: torch.empty(v.shape, dtype=v.dtype, device=self.device) for k, v in host.items()}
                     for _ in range(2)]
        self.copy_stream = torch.cuda.Stream(self.device)
        self.copied = [torch.cuda.Event() for _ in range(2)]
        self.released = [torch.cuda.Event() for _ in range(2)]
        self.stream = stream

    def _compute_stream(self):
        return torch.cuda.current_stream(self.device) if self.stream is None else self.stream

    def prefetch(self, slot, host):
        cs = self.copy_stream
        cs.wait_event(self.released[slot])  # a never-recorded event is already complete
        with torch.cuda.stream(cs):
            for k, v in host.items():
                self.bufs[slot][k].copy_(v, non_blocking=True)
        self.copied[slot].record(cs)

    def acquire(self, slot):
        self._compute_stream().wait_event(self.copied[slot])
        return self.bufs[slot]

    def release(self, slot):
        self.released[slot].record(self._compute_stream())


def score_calibrate_loss(h, W, targets, logp_old, r_bf16, adv, mask, coef, gran, eps_low, eps_high,
                         opts=None, buffers=None, stream=None):
    """One pass of the whole hot path through the C ABI, in order:
    quantize(h), quantize(W), token_logprobs (+ ratios), calibrate_clip_bounds,
    clipped_surrogate with the new bounds (and the calibration's count of valid
    tokens, so the surrogate makes no counting pass).  Returns the buffers
    object whose fields hold every output (device-resident)."""
    T, H = h.shape
    V = W.shape[0]
    b = buffers or StepBuffers(T, H, V, gran, h.device)
    quantize(h, gran, ROLE_ACT, b.h_codes, b.h_scales, b.q_ws, stream)
    quantize(W, gran, ROLE_WEIGHT, b.w_codes, b.w_scales, b.q_ws, stream)
    token_logprobs(b.h_codes, b.h_scales, b.w_codes, b.w_scales, gran, targets, logp_old,
                   workspace=b.lp_ws, out={"logp": b.logp, "lse": b.lse, "ratio": b.ratio}, stream=stream)
    calibrate_clip_bounds(b.ratio, r_bf16, adv, mask, coef, eps_low, eps_high, opts, b.cal_res,
                          b.cal_ws, stream)
    clipped_surrogate(b.ratio, adv, mask, None, bounds=bounds_view(b.cal_res), stats=b.stats,
                      workspace=b.sur_ws, out={"grad": b.grad, "clip_mask": b.clip_mask}, stream=stream,
                      n_valid=n_valid_view(b.cal_res))
    return b
