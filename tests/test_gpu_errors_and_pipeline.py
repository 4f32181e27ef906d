"""GPU: error reporting through the C ABI, the bounded-wait timeout path, and the
whole hot path in one call sequence (properties that hold at any size)."""

import ctypes
import dataclasses

import numpy as np
import pytest
import torch

from oracle import calibrate as OC
from oracle import quantize as OQ
from oracle import surrogate as OS
from paper_2609_22870_gb300 import synth
from tests.gpu_helpers import oracle_logprobs_rows, sample_rows

pytestmark = pytest.mark.gpu


def test_host_detected_errors(cuda_lib):
    api = cuda_lib
    x = torch.zeros(4, 200, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(api.Fp8rlError) as e:
        api.quantize(x[:, :192], api.GRAN_BLOCK, api.ROLE_ACT)  # 192 % 128 != 0
    assert e.value.status == api.ESHAPE
    st = api.lib.fp8rl_quantize(None, 4, 128, 128, 0, 0, None, None, None, 0, None)
    assert st == api.EINVAL
    buf = torch.zeros(4 * 136 + 8, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(4 * 128, dtype=torch.uint8, device="cuda")
    sc = torch.empty(4, dtype=torch.float32, device="cuda")
    st = api.lib.fp8rl_quantize(ctypes.c_void_p(buf.data_ptr() + 2), 4, 128, 136, 1, 0,
                                ctypes.c_void_p(codes.data_ptr()), ctypes.c_void_p(sc.data_ptr()),
                                None, 0, None)
    assert st == api.EALIGN
    st = api.lib.fp8rl_quantize(ctypes.c_void_p(buf.data_ptr()), 4, 128, 136, 0, 0,
                                ctypes.c_void_p(codes.data_ptr()), ctypes.c_void_p(sc.data_ptr()),
                                None, 0, None)
    assert st == api.EWORKSPACE
    api.check()


def test_bad_target_flags_device_error_and_nan(cuda_lib):
    api = cuda_lib
    h = synth.normal_bf16(130, 128, 1.0, 1, "cuda")
    W = synth.normal_bf16(300, 128, 0.02, 2, "cuda")
    y = torch.randint(0, 300, (130,), dtype=torch.int32, device="cuda")
    y[7] = 300
    y[9] = -1
    hc, hs = api.quantize(h, 0)
    wc, ws = api.quantize(W, 0, api.ROLE_WEIGHT)
    out = api.token_logprobs(hc, hs, wc, ws, 0, y)
    assert api.check_status() == api.EDEVICE
    lp = out["logp"].cpu().numpy()
    assert np.isnan(lp[7]) and np.isnan(lp[9]) and np.all(np.isfinite(np.delete(lp, [7, 9])))
    api.check()  # the status word was cleared


def test_non_finite_inputs_flag(cuda_lib):
    api = cuda_lib
    x = torch.zeros(3, 128, dtype=torch.bfloat16, device="cuda")
    x[1, 5] = float("inf")
    api.quantize(x, api.GRAN_BLOCK, api.ROLE_ACT)
    assert api.check_status() == api.EDEVICE
    r = torch.ones(10, device="cuda")
    r[3] = -1.0
    api.calibrate_clip_bounds(r, torch.ones(10, device="cuda"), -torch.ones(10, device="cuda"), None,
                              None, 0.2, 0.2)
    assert api.check_status() == api.EDEVICE
    api.check()


def test_bounded_wait_expires_and_context_survives(cuda_lib):
    api = cuda_lib
    api.wait_selftest(2_000_000)  # 2 ms; nothing signals the barrier
    assert api.check_status() == api.ETIMEOUT
    x = synth.normal_bf16(8, 128, 1.0, 3, "cuda")
    codes, scales = api.quantize(x, api.GRAN_ROWWISE)
    api.check()
    ref_c, _ = OQ.quantize(x.float().cpu().numpy(), OQ.ROWWISE)
    assert np.array_equal(codes.cpu().numpy(), ref_c)


@pytest.mark.parametrize("name,T,H,V", [("grpo_8b", 1100, 512, 5000), ("dapo_32b", 700, 640, 3000)])
def test_pipeline_small(cuda_lib, name, T, H, V):
    """score_calibrate_loss end to end at a size the oracle scores in full."""
    api = cuda_lib
    w = synth.scaled(synth.WORKLOADS[name], T=T, H=H, V=V)
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    adv, mask = synth.rollout(w)
    ref_lp, _, _ = oracle_logprobs_rows(h, W, w.gran, y, np.arange(w.T))
    noise = synth.old_policy_noise(w).numpy()
    logp_old = (ref_lp + noise).astype(np.float32)        # old policy near the BF16 scorer
    r_bf16 = np.exp(-noise).astype(np.float32)
    coef = np.exp(logp_old).astype(np.float32)
    b = api.score_calibrate_loss(h, W, y, torch.from_numpy(logp_old).cuda(), torch.from_numpy(r_bf16).cuda(),
                                 adv.cuda(), mask.cuda(), torch.from_numpy(coef).cuda(), w.gran,
                                 w.eps_low, w.eps_high)
    api.check()
    assert np.max(np.abs(b.logp.cpu().numpy() - ref_lp)) <= 2e-3
    res = api.read_calib_result(b.cal_res)
    st = api.read_clip_stats(b.stats)
    _pipeline_properties(res, st, b, adv.numpy(), mask.numpy(), r_bf16, w)


def test_pipeline_dapo_filter_with_forced_all_equal_group(cuda_lib):
    """DAPO workload with one group forced to all-equal rewards: the dynamic-
    sampling filter masks it, and no stage counts, clips or differentiates it."""
    api = cuda_lib
    w = dataclasses.replace(synth.WORKLOADS["dapo_32b"], name="dapo_forced", T=3 * 16 * 32, H=640, V=3000,
                            prompts=3, resp_len=32)
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    adv, mask = synth.rollout(w, force_equal_prompt=1)
    forced = np.zeros(w.T, bool)
    forced[16 * 32: 2 * 16 * 32] = True
    assert not mask.numpy()[forced].any()
    ref_lp, _, _ = oracle_logprobs_rows(h, W, w.gran, y, np.arange(w.T))
    noise = synth.old_policy_noise(w).numpy()
    logp_old = (ref_lp + noise).astype(np.float32)
    r_bf16 = np.exp(-noise).astype(np.float32)
    coef = np.exp(logp_old).astype(np.float32)
    b = api.score_calibrate_loss(h, W, y, torch.from_numpy(logp_old).cuda(), torch.from_numpy(r_bf16).cuda(),
                                 adv.cuda(), mask.cuda(), torch.from_numpy(coef).cuda(), w.gran,
                                 w.eps_low, w.eps_high)
    api.check()
    res = api.read_calib_result(b.cal_res)
    st = api.read_clip_stats(b.stats)
    _pipeline_properties(res, st, b, adv.numpy(), mask.numpy(), r_bf16, w)
    assert st["n_valid"] == int(mask.numpy().sum())
    assert not b.clip_mask.cpu().numpy()[forced].any()
    assert not b.grad.cpu().numpy()[forced].any()


def _pipeline_properties(res, st, b, adv, mask, r_bf16, w):
    r = b.ratio.cpu().numpy()
    neg = (mask != 0) & (adv < 0)
    pos = (mask != 0) & (adv > 0)
    c_lo, c_hi = OC.reference_bounds(w.eps_low, w.eps_high)
    assert res["n_neg"] == neg.sum() and res["n_pos"] == pos.sum()
    assert res["k_bf16"] == int(np.sum(neg & (r_bf16 <= c_lo)))
    assert res["k_fp8"] == int(np.sum(neg & (r <= np.float32(res["lo_star"]))))
    assert 0.5 <= res["lo_star"] <= 0.9 and 1.2 <= res["hi_star"] <= 2.0
    # new bounds = SmoothUpdate from no previous bound = searched bounds
    assert res["lo_new"] == res["lo_star"] and res["hi_new"] == res["hi_star"]
    # the loss used exactly these bounds
    assert st["lo"] == res["lo_new"] and st["hi"] == res["hi_new"]
    cm = b.clip_mask.cpu().numpy()
    assert np.array_equal((cm & 1) != 0, pos & (r >= np.float32(res["hi_new"])))
    assert np.array_equal((cm & 2) != 0, neg & (r <= np.float32(res["lo_new"])))


@pytest.mark.parametrize("name", ["grpo_8b", "dapo_32b", "long_8b"])
def test_pipeline_full_size(cuda_lib, name):
    """The whole path at the full configurations: logp on sampled rows against
    the oracle (the scoring tests check 1024+ rows per workload), every stage
    by the properties it must satisfy, and calibration and the loss bit for bit
    against the oracle run on the pipeline's own ratios."""
    api = cuda_lib
    w = synth.WORKLOADS[name]
    h, W, y = synth.hidden_states(w, "cuda"), synth.lm_head_weight(w, "cuda"), synth.targets(w, "cuda")
    adv, mask = synth.rollout(w)
    noise = synth.old_policy_noise(w)
    logp_old = torch.full((w.T,), -float(np.log(w.V))) + noise
    r_bf16 = torch.exp(-noise)
    coef = torch.exp(logp_old)
    b = api.score_calibrate_loss(h, W, y, logp_old.float().cuda(), r_bf16.float().cuda(), adv.cuda(),
                                 mask.cuda(), coef.float().cuda(), w.gran, w.eps_low, w.eps_high)
    api.check()
    rows = sample_rows(w.T, 16, 9)
    ref_lp, _, _ = oracle_logprobs_rows(h, W, w.gran, y, rows)
    assert np.max(np.abs(b.logp.cpu().numpy()[rows] - ref_lp)) <= 2e-3
    res = api.read_calib_result(b.cal_res)
    st = api.read_clip_stats(b.stats)
    _pipeline_properties(res, st, b, adv.numpy(), mask.numpy(), r_bf16.float().numpy(), w)
    # Calibration and the loss on the pipeline's own FP8 ratios: the oracle,
    # given the same ratios, must select the same bounds bit for bit (every
    # count and fixed-point sum too), and its surrogate with those bounds must
    # give the same clip mask, counts and fractions, the loss within 1e-4 and
    # the gradient within 1e-6.
    r = b.ratio.cpu().numpy()
    a_np, m_np = adv.numpy(), mask.numpy()
    ref = OC.calibrate_clip_bounds(r, r_bf16.float().numpy(), a_np, m_np, coef.float().numpy(),
                                   w.eps_low, w.eps_high)
    for k in ("lo_star", "hi_star", "lo_new", "hi_new", "c_lo", "c_hi"):
        assert np.float32(res[k]) == ref[k], (k, res[k], ref[k])
    for k in ("n_neg", "n_pos", "k_bf16", "k_fp8", "flags", "shift", "sum_pos_bf16", "sum_neg_bf16",
              "sum_neg_fp8", "sum_pos_fp8"):
        assert res[k] == ref[k], (k, res[k], ref[k])
    sref = OS.clipped_surrogate(r, a_np, m_np, None, ref["lo_new"], ref["hi_new"])
    assert np.array_equal(b.clip_mask.cpu().numpy(), sref["clip_mask"])
    for k in ("n_valid", "n_pos", "n_neg", "clipped_pos", "clipped_neg", "clip_frac_pos", "clip_frac_neg",
              "clip_frac"):
        assert st[k] == sref[k], (k, st[k], sref[k])
    scale = max(abs(sref["loss"]), np.sum(np.abs(sref["terms"])) / max(1, sref["n_valid"]))
    assert abs(st["loss"] - sref["loss"]) <= 1e-4 * scale
    g = b.grad.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(g - sref["grad"]) <= 1e-6 * np.abs(sref["grad"]) + 1e-30)


def test_prefetched_steps_match_direct_steps(cuda_lib):
    """Steps fed by the double-buffered host prefetcher (copies of step i + 1
    overlapping step i on a side stream) give the same results as direct
    steps: the copies are ordered before their use and after the slot's
    previous user."""
    api = cuda_lib
    w = synth.scaled(synth.WORKLOADS["grpo_8b"], T=4096, H=512, V=3000, name="pf")
    W = synth.lm_head_weight(w, "cuda")
    hosts = []
    for k in range(3):  # three different batches
        wk = synth.scaled(synth.WORKLOADS["grpo_8b"], T=4096, H=512, V=3000, name=f"pf{k}")
        wk = dataclasses.replace(wk, seed=100 + k)
        adv, mask = synth.rollout(wk)
        noise = synth.old_policy_noise(wk)
        lpo = (torch.full((w.T,), -8.0) + noise).float()
        hosts.append({"h": synth.hidden_states(wk, "cpu").pin_memory(), "y": synth.targets(wk, "cpu").pin_memory(),
                      "logp_old": lpo.pin_memory(), "r_bf16": torch.exp(-noise).float().pin_memory(),
                      "adv": adv.pin_memory(), "mask": mask.pin_memory(),
                      "coef": torch.exp(lpo).pin_memory()})
    stream = torch.cuda.current_stream()
    direct = []
    for hb in hosts:
        d = {k: v.cuda() for k, v in hb.items()}
        b = api.score_calibrate_loss(d["h"], W, d["y"], d["logp_old"], d["r_bf16"], d["adv"], d["mask"],
                                     d["coef"], w.gran, w.eps_low, w.eps_high)
        api.check()
        direct.append((api.read_calib_result(b.cal_res), b.grad.cpu().clone()))
    pf = api.HostBatchPrefetcher(hosts[0], "cuda", stream)
    b = api.StepBuffers(w.T, w.H, w.V, w.gran, "cuda")
    got = []
    pf.prefetch(0, hosts[0])
    for i in range(3):
        d = pf.acquire(i % 2)
        if i + 1 < 3:
            pf.prefetch((i + 1) % 2, hosts[i + 1])
        api.score_calibrate_loss(d["h"], W, d["y"], d["logp_old"], d["r_bf16"], d["adv"], d["mask"], d["coef"],
                                 w.gran, w.eps_low, w.eps_high, None, b, stream)
        pf.release(i % 2)
        api.check()
        got.append((api.read_calib_result(b.cal_res), b.grad.cpu().clone()))
    for (r0, g0), (r1, g1) in zip(direct, got):
        assert r0 == r1
        assert torch.equal(g0, g1)
