"""GPU: scoring without a caller workspace (fp8rl_token_logprobs_noalloc).

Some callers may not allocate device memory at the moment they score tokens:
serving loops and other hot paths that forbid allocation there (cudaMalloc and
cudaFree can synchronise the whole device), or processes whose device memory
is all reserved up front by another allocator.  They cannot hand
fp8rl_token_logprobs a workspace, so the no-alloc entry point uses a fixed
array inside the library instead.  These tests call it directly through the C
ABI, twice in a row with different shapes, and check its log-probs against
the oracle (within the 2e-3 log-prob tolerance of the other GPU tests) and
its log-probs, logsumexps and ratios bit for bit against fp8rl_token_logprobs
with a normal workspace (the same kernels run on the same inputs).

This file is collected last so that a run stopping at its first failure has
already run every other test.
"""

import ctypes

import numpy as np
import pytest
import torch

from paper_2609_22870_gb300 import synth
from tests.gpu_helpers import oracle_logprobs_rows

pytestmark = pytest.mark.gpu
TOL = 2e-3


def _fn(api):
    fn = api.lib.fp8rl_token_logprobs_noalloc
    p, i64 = ctypes.c_void_p, ctypes.c_int64
    fn.restype = ctypes.c_int
    fn.argtypes = [p, p, p, p, ctypes.c_int, i64, i64, i64, p, p, p, p, p, p]
    return fn


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


@pytest.mark.parametrize("gran", [0, 1, 2])
def test_noalloc_matches_oracle_and_workspace_call_two_calls(cuda_lib, gran):
    api = cuda_lib
    fn = _fn(api)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call, (T, H, V, seed) in enumerate([(300, 256, 5000, 11), (1200, 512, 3000, 12)]):
        h = synth.normal_bf16(T, H, 1.0, seed, "cuda")
        W = synth.normal_bf16(V, H, 0.02, seed + 1, "cuda")
        g = torch.Generator().manual_seed(seed)
        y = torch.randint(0, V, (T,), generator=g).to(torch.int32).cuda()
        logp_old = (torch.randn(T, generator=g) - float(np.log(V))).float().cuda()
        hc, hs = api.quantize(h, gran, api.ROLE_ACT)
        wc, ws = api.quantize(W, gran, api.ROLE_WEIGHT)
        logp, lse, ratio = (torch.full((T,), float("nan"), device="cuda") for _ in range(3))
        st = fn(_ptr(hc), _ptr(hs), _ptr(wc), _ptr(ws), gran, T, H, V, _ptr(y), _ptr(logp_old),
                _ptr(logp), _ptr(lse), _ptr(ratio), stream)
        assert st == api.OK, (call, st)
        api.check()
        # against the oracle, which quantises the same bf16 inputs itself
        ref_lp, ref_lse, _ = oracle_logprobs_rows(h, W, gran, y, np.arange(T))
        assert np.max(np.abs(logp.cpu().numpy() - ref_lp)) <= TOL, call
        assert np.max(np.abs(lse.cpu().numpy() - ref_lse)) <= TOL, call
        # and bit for bit against the call with a caller workspace
        ref = api.token_logprobs(hc, hs, wc, ws, gran, y, logp_old)
        api.check()
        for k, got in (("logp", logp), ("lse", lse), ("ratio", ratio)):
            assert torch.equal(got, ref[k]), (call, k)


def test_noalloc_refuses_shapes_beyond_its_scratch(cuda_lib):
    api = cuda_lib
    fn = _fn(api)
    T, H, V = 4096, 128, 151936  # needs ~39 MB of scratch
    assert api.token_logprobs_workspace_size(T, H, V, 2) > (16 << 20)
    dummy = torch.zeros(16, dtype=torch.uint8, device="cuda")
    st = fn(_ptr(dummy), _ptr(dummy), _ptr(dummy), _ptr(dummy), 2, T, H, V, _ptr(dummy), None,
            _ptr(dummy), None, None, None)
    assert st == api.EWORKSPACE
