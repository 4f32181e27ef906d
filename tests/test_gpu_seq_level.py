"""GPU parity: sequence-level ratio clipping (one geometric-mean ratio per
response, clipped like a token ratio; the response-level trust region of the
related-work discussion, §6).

The sequence ratio s_i is float32 on both sides; the kernel's exponent sum is
exact on the 2^-32 grid, so its s_i may differ from the oracle's by one float32
ulp in rare cases.  Where both agree the clip bits are compared bit-exactly;
everywhere the kernel's bits must follow the clip rule applied to its own s_i.
The gradient is the float64 quotient rounded once to float32 (within 2^-24
relative of the oracle's float64 value); the loss within 1e-6 of the mean
|term|.
"""

import numpy as np
import pytest
import torch

from oracle import surrogate as OS
from paper_2609_22870_gb300 import synth

pytestmark = pytest.mark.gpu


def _seq_ids(T, n_seq, seed, contiguous=True):
    g = torch.Generator().manual_seed(seed + 11)
    if contiguous:  # packed responses of random lengths
        cuts = torch.sort(torch.randint(0, T + 1, (max(n_seq - 1, 0),), generator=g)).values
        sid = torch.bucketize(torch.arange(T), cuts, right=True)
    else:
        sid = torch.randint(0, max(n_seq, 1), (T,), generator=g)
    return sid.to(torch.int32)


def _inputs(T, n_seq, seed, contiguous=True, seq_sigma=0.2, tok_sigma=0.3):
    """logp ~ N(-3, 1); logp_old = logp - (b_i + e_t) with a per-response
    drift b_i and per-token noise e_t, so the response ratios straddle the
    bounds."""
    g = torch.Generator().manual_seed(seed)
    sid = _seq_ids(T, n_seq, seed, contiguous)
    lp = (torch.randn(T, generator=g) - 3.0).float()
    b = torch.randn(max(n_seq, 1), generator=g) * seq_sigma
    e = torch.randn(T, generator=g) * tok_sigma
    lpo = (lp - (b[sid.long()] + e)).float() if T else lp.clone()
    A = torch.randn(max(n_seq, 1), generator=g).float()[:n_seq]
    if n_seq > 4:
        A[::7] = 0
    mask = (torch.rand(T, generator=g) < 0.85).to(torch.uint8)
    return lp, lpo, A, mask, sid


def _rule(s, A, n_valid, lo, hi):
    up = (n_valid > 0) & (A > 0) & (s >= np.float32(hi))
    dn = (n_valid > 0) & (A < 0) & (s <= np.float32(lo))
    return (up * OS.CLIP_HI + dn * OS.CLIP_LO).astype(np.uint8)


def _check(api, lp, lpo, A, mask, sid, lo=0.8, hi=1.2, bounds=None):
    n_seq = A.numel()
    m = None if mask is None else mask.cuda()
    out = api.seq_level_clipped_surrogate(lp.cuda(), lpo.cuda(), A.cuda(), sid.cuda(), mask=m, lo=lo, hi=hi,
                                          bounds=bounds)
    api.check()
    st = api.read_clip_stats(out["stats"])
    L, H = (float(bounds[0]), float(bounds[1])) if bounds is not None else (lo, hi)
    ref = OS.seq_level_clipped_surrogate(lp.numpy(), lpo.numpy(), A.numpy(),
                                         None if mask is None else mask.numpy(), sid.numpy(), n_seq, L, H)
    s = out["seq_ratio"].cpu().numpy()
    s_ref = ref["seq_ratio32"]
    assert np.all(np.abs(s.view(np.int32).astype(np.int64) - s_ref.view(np.int32).astype(np.int64)) <= 1)
    same = s == s_ref
    cm = out["seq_clip"].cpu().numpy()
    assert np.array_equal(cm[same], ref["seq_clip"][same])
    assert np.array_equal(cm, _rule(s, A.numpy(), ref["seq_valid_tokens"], L, H))
    for k in ("n_valid", "n_seq_valid", "n_pos", "n_neg"):
        assert st[k] == ref[k], k
    if same.all():
        assert st["clipped_pos"] == ref["clipped_pos"] and st["clipped_neg"] == ref["clipped_neg"]
        for k in ("clip_frac_pos", "clip_frac_neg", "clip_frac"):
            assert st[k] == ref[k], k
    # the fractions the library reports are those of its own counts
    assert st["clip_frac_pos"] == (st["clipped_pos"] / st["n_pos"] if st["n_pos"] else 0.0)
    assert st["clip_frac_neg"] == (st["clipped_neg"] / st["n_neg"] if st["n_neg"] else 0.0)
    S = st["n_seq_valid"]
    assert st["clip_frac"] == ((st["clipped_pos"] + st["clipped_neg"]) / S if S else 0.0)
    scale = max(abs(ref["loss"]), np.sum(np.abs(ref["seq_terms"])) / max(1, ref["n_seq_valid"]), 1e-300)
    assert abs(st["loss"] - ref["loss"]) <= 1e-6 * scale
    assert st["flags"] == (0 if ref["n_valid"] else 1)
    g = out["grad"].cpu().numpy().astype(np.float64)
    tok_same = same[sid.numpy()] if sid.numel() else np.zeros(0, bool)
    gr = ref["grad"]
    assert np.all(np.abs(g - gr)[tok_same] <= 2.0 ** -23 * np.abs(gr)[tok_same])
    assert np.all(g[tok_same & (gr == 0)] == 0)
    return st, out, ref


@pytest.mark.parametrize("T,n_seq", [(1, 1), (37, 3), (1000, 40), (4099, 32), (65539, 128), (131072, 8)])
@pytest.mark.parametrize("contiguous", [True, False])
def test_seq_level_parity(cuda_lib, T, n_seq, contiguous):
    st, _, ref = _check(cuda_lib, *_inputs(T, n_seq, T + 3 * n_seq, contiguous))
    if n_seq >= 32:  # the inputs clip responses on both sides
        assert ref["clipped_pos"] > 0 and ref["clipped_neg"] > 0


def test_seq_level_grpo_layout(cuda_lib):
    """The grpo_8b batch layout: 4 prompts x 8 responses x 512 slots, GRPO
    group advantages, length mask U[64, 512]; bounds from a device buffer."""
    w = synth.WORKLOADS["grpo_8b"]
    adv, mask = synth.rollout(w)
    n_seq = w.prompts * w.group
    sid = (torch.arange(w.T) // w.resp_len).to(torch.int32)
    A = adv.reshape(n_seq, w.resp_len)[:, 0].contiguous()
    g = torch.Generator().manual_seed(41)
    lp = (torch.randn(w.T, generator=g) - 3.0).float()
    drift = torch.randn(n_seq, generator=g) * 0.15
    lpo = (lp - drift[sid.long()] - torch.randn(w.T, generator=g) * 0.05).float()
    b = torch.tensor([0.9, 1.1], dtype=torch.float32, device="cuda")
    _check(cuda_lib, lp, lpo, A, mask, sid, bounds=b)


def test_seq_level_ties_at_the_bounds(cuda_lib):
    """Responses whose every token has d = fl32(log H) (or fl32(log L)) have
    s_i = H (or L) exactly: clipped at equality for A > 0 (A < 0)."""
    H32, L32 = np.float32(1.2), np.float32(0.8)
    dH, dL = np.float32(np.log(np.float64(H32))), np.float32(np.log(np.float64(L32)))
    assert np.float32(np.exp(np.float64(dH))) == H32 and np.float32(np.exp(np.float64(dL))) == L32
    n_seq, per = 8, 50
    kind = np.repeat(np.array([0, 1, 0, 1, 0, 1, 2, 2]), per)  # 0: d = dH, 1: d = dL, 2: d = 0
    lp = np.where(kind == 0, 0.0, np.where(kind == 1, dL, -1.0)).astype(np.float32)
    lpo = np.where(kind == 0, -dH, np.where(kind == 1, 0.0, -1.0)).astype(np.float32)
    d = lp - lpo  # the float32 difference the path forms
    assert np.all(d[kind == 0] == dH) and np.all(d[kind == 1] == dL) and np.all(d[kind == 2] == 0)
    sid = torch.from_numpy(np.repeat(np.arange(n_seq), per).astype(np.int32))
    A = torch.tensor([1.0, -1.0, -1.0, 1.0, 0.0, 0.0, 1.0, -1.0])
    _, out, _ = _check(cuda_lib, torch.from_numpy(lp), torch.from_numpy(lpo), A, None, sid)
    s = out["seq_ratio"].cpu().numpy()
    assert np.all(s[[0, 2, 4]] == H32) and np.all(s[[1, 3, 5]] == L32) and np.all(s[6:] == 1)
    assert list(out["seq_clip"].cpu().numpy()) == [OS.CLIP_HI, OS.CLIP_LO, 0, 0, 0, 0, 0, 0]


def test_seq_level_empty_and_nullable(cuda_lib):
    api = cuda_lib
    e = torch.empty(0, device="cuda")
    out = api.seq_level_clipped_surrogate(e, e, e, torch.empty(0, dtype=torch.int32, device="cuda"))
    api.check()
    st = api.read_clip_stats(out["stats"])
    assert st["loss"] == 0 and st["n_valid"] == 0 and st["n_seq_valid"] == 0 and st["flags"] == 1
    # sequences but no tokens; then every token masked
    A = torch.ones(5, device="cuda")
    out = api.seq_level_clipped_surrogate(e, e, A, torch.empty(0, dtype=torch.int32, device="cuda"))
    api.check()
    assert not out["seq_ratio"].any() and not out["seq_clip"].any()
    lp, lpo, A, _, sid = _inputs(500, 9, 5)
    st, _, _ = _check(api, lp, lpo, A, torch.zeros(500, dtype=torch.uint8), sid)
    assert st["loss"] == 0 and st["n_seq_valid"] == 0 and st["flags"] == 1
    _check(api, lp, lpo, A, None, sid)  # no mask: every token valid


def test_seq_level_unaligned_and_ragged(cuda_lib):
    """Views starting one element in (no 16-byte alignment) take the scalar path."""
    lp, lpo, A, mask, sid = _inputs(3001, 17, 8)
    api = cuda_lib
    dl, dlo, dm, ds = (t.cuda() for t in (lp, lpo, mask, sid))
    out = api.seq_level_clipped_surrogate(dl[1:], dlo[1:], A.cuda(), ds[1:], mask=dm[1:])
    api.check()
    ref = OS.seq_level_clipped_surrogate(lp[1:].numpy(), lpo[1:].numpy(), A.numpy(), mask[1:].numpy(),
                                         sid[1:].numpy(), 17, 0.8, 1.2)
    st = api.read_clip_stats(out["stats"])
    assert st["n_valid"] == ref["n_valid"] and st["n_seq_valid"] == ref["n_seq_valid"]
    g = out["grad"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(g - ref["grad"]) <= 2.0 ** -23 * np.abs(ref["grad"]))


def test_seq_level_deterministic_and_order_free(cuda_lib):
    """Integer exponent sums: the same result for any token order."""
    lp, lpo, A, mask, sid = _inputs(200000, 300, 12, contiguous=False)
    api = cuda_lib
    a = api.seq_level_clipped_surrogate(lp.cuda(), lpo.cuda(), A.cuda(), sid.cuda(), mask=mask.cuda())
    p = torch.randperm(200000, generator=torch.Generator().manual_seed(3))
    b = api.seq_level_clipped_surrogate(lp[p].cuda(), lpo[p].cuda(), A.cuda(), sid[p].cuda(),
                                        mask=mask[p].cuda())
    api.check()
    assert torch.equal(a["seq_ratio"], b["seq_ratio"]) and torch.equal(a["seq_clip"], b["seq_clip"])
    assert torch.equal(a["grad"][p.cuda()], b["grad"])
    sa, sb = api.read_clip_stats(a["stats"]), api.read_clip_stats(b["stats"])
    assert sa["loss"] == sb["loss"]


def test_seq_level_bad_input_flagged(cuda_lib):
    api = cuda_lib
    lp, lpo, A, mask, sid = (t.cuda() for t in _inputs(300, 5, 6))
    bad = sid.clone()
    bad[17] = 5  # n_seq = 5: out of range
    api.seq_level_clipped_surrogate(lp, lpo, A, bad, mask=mask)
    assert api.check_status() == api.EDEVICE
    far = lp.clone()
    far[3] = lpo[3] + 200.0  # |d| > 128 on a valid token
    api.seq_level_clipped_surrogate(far, lpo, A, sid, mask=None)
    assert api.check_status() == api.EDEVICE
    nan = lp.clone()
    nan[4] = float("nan")
    api.seq_level_clipped_surrogate(nan, lpo, A, sid, mask=None)
    assert api.check_status() == api.EDEVICE
    m = torch.ones(300, dtype=torch.uint8, device="cuda")
    m[3] = 0  # the same far token, masked: no flag
    api.seq_level_clipped_surrogate(far, lpo, A, sid, mask=m)
    assert api.check_status() == 0
    with pytest.raises(ValueError):
        api.seq_level_clipped_surrogate(lp, lpo[:10], A, sid)


def test_seq_level_stress_size_sampled(cuda_lib):
    """2^26 tokens in responses of 512 (the stress size of the kernel bench,
    halved): every count exact, and sampled responses against the oracle run on
    their own tokens (their s_i and clip bits do not depend on the others; the
    gradient scales by S)."""
    api = cuda_lib
    T, per = 1 << 26, 512
    n_seq = T // per
    dev = torch.device("cuda")
    g = torch.Generator(device=dev)
    g.manual_seed(77)
    sid = (torch.arange(T, device=dev, dtype=torch.int64) // per).to(torch.int32)
    lp = torch.randn(T, generator=g, device=dev) - 3.0
    drift = torch.randn(n_seq, generator=g, device=dev) * 0.2
    lpo = lp - drift[sid.long()] - torch.randn(T, generator=g, device=dev) * 0.3
    A = torch.randn(n_seq, generator=g, device=dev)
    mask = (torch.rand(T, generator=g, device=dev) < 0.9).to(torch.uint8)
    out = api.seq_level_clipped_surrogate(lp, lpo, A, sid, mask=mask)
    api.check()
    st = api.read_clip_stats(out["stats"])
    assert st["n_valid"] == int(mask.sum()) and st["n_seq_valid"] == n_seq
    pick = np.random.default_rng(5).choice(n_seq, 48, replace=False)
    rows = torch.from_numpy(np.concatenate([np.arange(i * per, (i + 1) * per) for i in pick])).to(dev)
    sub_sid = torch.from_numpy(np.repeat(np.arange(48), per).astype(np.int32))
    ref = OS.seq_level_clipped_surrogate(lp[rows].cpu().numpy(), lpo[rows].cpu().numpy(),
                                         A[torch.from_numpy(pick).to(dev)].cpu().numpy(),
                                         mask[rows].cpu().numpy(), sub_sid.numpy(), 48, 0.8, 1.2)
    s = out["seq_ratio"][torch.from_numpy(pick).to(dev)].cpu().numpy()
    same = s == ref["seq_ratio32"]
    assert np.all(np.abs(s.view(np.int32).astype(np.int64) - ref["seq_ratio32"].view(np.int32)) <= 1)
    assert np.array_equal(out["seq_clip"][torch.from_numpy(pick).to(dev)].cpu().numpy()[same],
                          ref["seq_clip"][same])
    g_gpu = out["grad"][rows].cpu().numpy().astype(np.float64)
    g_ref = ref["grad"] * (48 / n_seq)  # the oracle's S is the sample's
    tok_same = same[sub_sid.numpy()]
    assert np.all(np.abs(g_gpu - g_ref)[tok_same] <= 1e-6 * np.abs(g_ref)[tok_same])
