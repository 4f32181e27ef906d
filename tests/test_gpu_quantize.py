"""GPU parity: E4M3 quantisation (Eq. 3) bit-exact against the oracle."""

import numpy as np
import pytest
import torch

from oracle import e4m3
from oracle import quantize as OQ
from paper_2609_22870_gb300 import synth
from tests.gpu_helpers import scales_natural

pytestmark = pytest.mark.gpu

CASES = [(OQ.TENSOR, OQ.ACT), (OQ.ROWWISE, OQ.ACT), (OQ.ROWWISE, OQ.WEIGHT),
         (OQ.BLOCK, OQ.ACT), (OQ.BLOCK, OQ.WEIGHT)]


def _input(rows, cols, seed, ld=None):
    x = synth.normal_bf16(rows, cols, 1.0, seed, "cuda").float()
    g = torch.Generator(device="cpu").manual_seed(seed)
    rowscale = torch.exp2(torch.randint(-20, 12, (rows, 1), generator=g).float()).cuda()
    x = x * rowscale
    if rows > 3:
        x[1] = 0.0                      # an all-zero row: S = 1
        x[2, : min(cols, 200)] = 0.0    # zero blocks
    x = x.to(torch.bfloat16)
    if ld is not None and ld > cols:
        big = torch.zeros(rows, ld, dtype=torch.bfloat16, device="cuda")
        big[:, :cols] = x
        x = big[:, :cols]
    return x


@pytest.mark.parametrize("gran,role", CASES)
@pytest.mark.parametrize("rows,cols,ld", [(1, 128, None), (7, 256, None), (129, 384, 512),
                                          (300, 512, None), (1000, 4096, None), (257, 5120, None)])
def test_quantize_bit_exact(cuda_lib, gran, role, rows, cols, ld):
    x = _input(rows, cols, rows * 31 + cols, ld)
    codes, scales = cuda_lib.quantize(x, gran, role)
    cuda_lib.check()
    ref_c, ref_s = OQ.quantize(x.float().cpu().numpy(), gran, role)
    assert np.array_equal(codes.cpu().numpy(), ref_c)
    assert np.array_equal(scales_natural(scales, rows, cols, gran, role), ref_s)


@pytest.mark.parametrize("gran", [OQ.ROWWISE])
def test_quantize_non_block_cols_multiple_of_16(cuda_lib, gran):
    x = _input(33, 48, 5)
    codes, scales = cuda_lib.quantize(x, gran, OQ.ACT)
    cuda_lib.check()
    ref_c, ref_s = OQ.quantize(x.float().cpu().numpy(), gran, OQ.ACT)
    assert np.array_equal(codes.cpu().numpy(), ref_c)
    assert np.array_equal(scales.cpu().numpy()[:33], ref_s)


@pytest.mark.parametrize("name", ["grpo_8b", "dapo_32b"])
@pytest.mark.parametrize("gran", [OQ.TENSOR, OQ.ROWWISE, OQ.BLOCK])
def test_quantize_full_size_lm_head_sampled(cuda_lib, name, gran):
    """Full Qwen-sized lm_head W (V = 151936): sampled 128-row strips bit-exact."""
    w = synth.WORKLOADS[name]
    W = synth.lm_head_weight(w, "cuda")
    codes, scales = cuda_lib.quantize(W, gran, OQ.WEIGHT)
    cuda_lib.check()
    V, H = W.shape
    rng = np.random.default_rng(0)
    strips = sorted(set(rng.choice(V // 128, 6, replace=False).tolist() + [0, (V - 1) // 128]))
    s_all = scales_natural(scales, V, H, gran, OQ.WEIGHT)
    if gran == OQ.TENSOR:
        amax = np.float32(0)
        for v0 in range(0, V, 8192):
            amax = max(amax, np.max(np.abs(W[v0:v0 + 8192].float().cpu().numpy())))
        s_ref = OQ.scale_from_amax(amax).reshape(1)
        assert np.array_equal(s_all, s_ref)
    for sb in strips:
        r0, r1 = sb * 128, min(V, sb * 128 + 128)
        xs = W[r0:r1].float().cpu().numpy()
        if gran == OQ.TENSOR:
            ref_c = OQ._encode_block(xs, s_ref[0])
        else:
            ref_c, ref_s = OQ.quantize(xs, gran, OQ.WEIGHT)
            got_s = s_all[r0:r1] if gran == OQ.ROWWISE else s_all[sb:sb + 1]
            assert np.array_equal(got_s, ref_s)
        assert np.array_equal(codes[r0:r1].cpu().numpy(), ref_c), (gran, sb)


@pytest.mark.parametrize("name", ["grpo_8b", "long_8b"])
def test_quantize_full_size_hidden_sampled(cuda_lib, name):
    w = synth.WORKLOADS[name]
    h = synth.hidden_states(w, "cuda")
    codes, scales = cuda_lib.quantize(h, OQ.BLOCK, OQ.ACT)
    cuda_lib.check()
    rows = np.array(sorted(set(np.random.default_rng(1).choice(w.T, 200, replace=False).tolist()
                               + [0, w.T - 1])))
    ref_c, ref_s = OQ.quantize(h[torch.as_tensor(rows).cuda()].float().cpu().numpy(), OQ.BLOCK, OQ.ACT)
    s_all = scales_natural(scales, w.T, w.H, OQ.BLOCK, OQ.ACT)
    assert np.array_equal(codes[torch.as_tensor(rows).cuda()].cpu().numpy(), ref_c)
    assert np.array_equal(s_all[rows], ref_s)


def _adversarial_bits(seed):
    """One 128-element row per positive finite bf16 amax (bit patterns
    0x0001 .. 0x7F7F, so every block scale S a bf16 block can have, from the
    subnormal range to 3.39e38 / 448), the other elements placed on bf16
    values next to E4M3 rounding midpoints times S, where the quotient's last
    bits decide the code, plus signed zeros."""
    rng = np.random.default_rng(seed)
    a_bits = np.arange(1, 0x7F80, dtype=np.uint32)
    n = a_bits.size
    amax = (a_bits << 16).view(np.float32)
    s = OQ.scale_from_amax(amax).astype(np.float64)
    vals = np.sort(np.unique(np.abs(e4m3.decode(np.arange(0, 0x7F, dtype=np.uint8)).astype(np.float64))))
    mids = (vals[:-1] + vals[1:]) / 2
    target = mids[rng.integers(0, mids.size, size=(n, 127))] * s[:, None]
    t = target.astype(np.float32).view(np.uint32)
    rb = (t + 0x7FFF + ((t >> 16) & 1)) >> 16                  # nearest bf16
    rb = rb.astype(np.int64) + rng.integers(-1, 2, size=rb.shape)  # and its neighbours
    rb = np.clip(rb, 0, a_bits[:, None].astype(np.int64))
    sign = rng.integers(0, 2, size=(n, 128)).astype(np.int64) << 15
    bits = np.empty((n, 128), dtype=np.int64)
    bits[:, 0] = a_bits
    bits[:, 1:] = rb
    bits |= sign
    bits[::3, 127] = 0x8000                                     # -0
    bits[1::3, 127] = 0x0000                                    # +0
    return bits.astype(np.uint16).view(np.int16)


@pytest.mark.parametrize("gran,role", CASES)
def test_quantize_every_bf16_scale_near_midpoints(cuda_lib, gran, role):
    """The division-free quotient against fl32(x / S) at every block scale
    and at the inputs most sensitive to its last bit."""
    bits = _adversarial_bits(7)
    x = torch.from_numpy(bits).view(torch.bfloat16).cuda()
    rows, cols = x.shape
    codes, scales = cuda_lib.quantize(x, gran, role)
    cuda_lib.check()
    ref_c, ref_s = OQ.quantize(x.float().cpu().numpy(), gran, role)
    assert np.array_equal(scales_natural(scales, rows, cols, gran, role), ref_s)
    got = codes.cpu().numpy()
    bad = np.argwhere(got != ref_c)
    assert bad.size == 0, (bad[:5], got[tuple(bad[0])], ref_c[tuple(bad[0])])


# ---- power-of-two (UE8M0) scales ----------------------------------------------

@pytest.mark.parametrize("gran,role", CASES)
@pytest.mark.parametrize("rows,cols,ld", [(7, 256, None), (129, 384, 512), (1000, 4096, None)])
def test_quantize_ue8m0_bit_exact(cuda_lib, gran, role, rows, cols, ld):
    x = _input(rows, cols, rows * 17 + cols, ld)
    codes, scales = cuda_lib.quantize(x, gran, role, ue8m0=True)
    cuda_lib.check()
    ref_c, ref_s = OQ.quantize(x.float().cpu().numpy(), gran, role, pow2=True)
    assert np.array_equal(codes.cpu().numpy(), ref_c)
    assert np.array_equal(scales_natural(scales, rows, cols, gran, role), ref_s)


@pytest.mark.parametrize("gran", [OQ.TENSOR, OQ.ROWWISE, OQ.BLOCK])
def test_logprobs_on_ue8m0_codes(cuda_lib, gran):
    """The scoring GEMM takes power-of-two scales like any other."""
    from oracle import logprobs as OL
    api = cuda_lib
    T, H, V = 300, 256, 1000
    h = synth.normal_bf16(T, H, 1.0, 61, "cuda")
    W = synth.normal_bf16(V, H, 0.05, 62, "cuda")
    y = torch.randint(0, V, (T,), generator=torch.Generator().manual_seed(63)).to(torch.int32).cuda()
    hc, hs = api.quantize(h, gran, api.ROLE_ACT, ue8m0=True)
    wc, ws = api.quantize(W, gran, api.ROLE_WEIGHT, ue8m0=True)
    out = api.token_logprobs(hc, hs, wc, ws, gran, y)
    api.check()
    hq, hsr = OQ.quantize(h.float().cpu().numpy(), gran, OQ.ACT, pow2=True)
    wq, wsr = OQ.quantize(W.float().cpu().numpy(), gran, OQ.WEIGHT, pow2=True)
    ref, _ = OL.token_logprobs(hq, hsr, wq, wsr, gran, y.cpu().numpy())
    assert np.max(np.abs(out["logp"].cpu().numpy() - ref)) <= 2e-3


@pytest.mark.parametrize("ue8m0", [False, True])
@pytest.mark.parametrize("gran,role", [(2, 0), (2, 1), (1, 0)])
def test_non_finite_block_shows_in_its_scale(cuda_lib, ue8m0, gran, role):
    """A NaN or inf input flags the call and leaves a non-finite scale for its
    own block (NaN stays NaN, inf stays inf, in both scale modes); every other
    block's scale is the oracle's."""
    api = cuda_lib
    rows, cols = 256, 384
    x = synth.normal_bf16(rows, cols, 1.0, 77, "cuda")
    x[3, 5] = float("nan")
    x[200, 300] = float("inf")
    codes, scales = api.quantize(x, gran, role, ue8m0=ue8m0)
    assert api.check_status() == api.EDEVICE
    got = scales_natural(scales, rows, cols, gran, role)
    if gran == 1:
        bad = {(3,): "nan", (200,): "inf"}
        idx = lambda r, c: (r,)  # noqa: E731
    elif role == 0:
        bad = {(3, 0): "nan", (200, 2): "inf"}
        idx = lambda r, c: (r, c // 128)  # noqa: E731
    else:
        bad = {(0, 0): "nan", (1, 2): "inf"}
        idx = lambda r, c: (r // 128, c // 128)  # noqa: E731
    for k, kind in bad.items():
        v = got[k]
        assert (np.isnan(v) if kind == "nan" else np.isposinf(v)), (k, v)
    clean = x.float().cpu().numpy()
    clean[3, 5] = 0.0
    clean[200, 300] = 0.0
    _, ref = OQ.quantize(clean, gran, role, pow2=ue8m0)
    keep = np.ones(ref.shape, bool)
    for k in bad:
        keep[k] = False
    # blocks without a bad element match (the zeroed ones may differ only if
    # the bad element was their maximum, which the mask above excludes)
    assert np.array_equal(got[keep], ref[keep])
