"""Benchmark: scored tokens/s of the FP8 log-prob + Calibrated-Clipping path.

One step = one pass of the whole hot path over one synthetic batch of the
8B-shaped GRPO workload (T = 16384 tokens, hidden 4096, vocab 151936, 1x128 /
128x128 block E4M3 scaling): quantise h, quantise W, FP8 GEMM with streaming
logsumexp + target gather, combine into log-probs and ratios, calibrate the
clip bounds, clipped surrogate with token-mean loss, clip counts and
dloss/dlogp.  Inputs are resident in HBM when the timed region starts (the W
codes alone, 622 MB, exceed L2, so no flush is needed); ``e2e`` repeats the
measurement with the per-step inputs in pinned host memory, copied in and the
result read back inside the timed region.

--impl reference times the CPU oracle on the host cores instead (bounded
samples of the same workload, extrapolated to a full step).
Multi-GPU (torchrun): every rank runs its own replica of the workload (weak
scaling, no collective on the data path); value = all tokens / max rank time.
"""

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "scored tokens/sec (FP8 logprob+calibrated-clip loss) at 8B shape; % FP8 peak, % HBM"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
FP8_OVER_BF16 = 4.5 / 2.25  # nominal dense FP8 / BF16 tensor rates
GRAN_NAMES = {0: "tensor", 1: "row", 2: "block"}

# DRAM bytes (read + write) per launch of the GEMM kernel on the default
# workload, from one ncu capture of this kernel source at that workload
# (dram__bytes_read.sum + dram__bytes_write.sum); reported only while the
# kernel sources (gemm.cu, gemm_epi.cuh) are the ones that were measured.
GEMM_TRAFFIC = {"workload": "grpo_8b", "bytes": 1.953e9, "gemm_sources_sha256_prefix": "1a921cc652e4e61e"}


def max_over_ranks(values, world, device="cpu"):
    """Per-rank timings -> their maxima over all ranks: a job of N replicas is as
    slow as its slowest rank.  One process per GPU with NCCL on GPUs; the same
    code runs over gloo on CPU in the tests."""
    if world <= 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.cpu()]


def whole_job_rate(units_per_rank, world, ms):
    """Units processed by all ranks per second, from the max-over-ranks time."""
    return world * units_per_rank / (ms * 1e-3)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def gemm_source_digest():
    """sha256 prefix over the GEMM kernel's sources (gemm.cu, then gemm_epi.cuh)."""
    import hashlib
    h = hashlib.sha256()
    for name in ("gemm.cu", "gemm_epi.cuh"):
        with open(os.path.join(ROOT, "paper_2609_22870_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def measured_gemm_traffic(w):
    if w.name == GEMM_TRAFFIC["workload"] and gemm_source_digest() == GEMM_TRAFFIC["gemm_sources_sha256_prefix"]:
        return GEMM_TRAFFIC["bytes"]
    return None


def workload_desc(w):
    lm = f", length mask U[{w.length_mask[0]},{w.length_mask[1]}]" if w.length_mask else ""
    flt = ", all-equal groups masked (DAPO filter)" if w.filter_equal_groups else ""
    return (f"{w.name}: T={w.T}, H={w.H}, V={w.V}, {GRAN_NAMES[w.gran]} E4M3 scaling, "
            f"{w.prompts}x{w.group} responses x {w.resp_len}, rewards Bern({w.reward_p}), "
            f"eps_low={w.eps_low}, eps_high={w.eps_high}{lm}{flt}")


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """SM clock and throttle reasons sampled during the timed regions.

    NVML is read through ctypes every ~5 ms (the GPU is found by its PCI bus
    id, so the sample is of the device this process runs on whatever its
    index); without NVML, nvidia-smi every 100 ms.  Reading clocks changes no
    GPU setting.  Sampling runs only inside ``with sampler.active():`` blocks,
    so idle gaps between timed regions do not dilute the median."""

    # NVML clocks-event (throttle) reason bits
    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown",
               0x4: "sw_power_cap"}

    def __init__(self, pci_bus_id, index):
        self.pci = pci_bus_id
        self.index = index
        self.sm, self.reasons = [], set()
        self.smax = None
        self.power_limit_w = None
        self.region = None
        self.by_region = {}  # region -> ([sm MHz], [power W])
        self._on = threading.Event()
        self._stop = threading.Event()
        self.src = None
        self.nvml = self._open_nvml()
        self.proc = None
        if self.nvml is not None:
            self.thread = threading.Thread(target=self._nvml_loop, daemon=True)
            self.thread.start()
            self.src = "nvml"

    def _open_nvml(self):
        import ctypes
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return None
            h = ctypes.c_void_p()
            ok = False
            if self.pci:
                ok = lib.nvmlDeviceGetHandleByPciBusId_v2(self.pci.encode(), ctypes.byref(h)) == 0
            if not ok and lib.nvmlDeviceGetHandleByIndex_v2(int(self.index), ctypes.byref(h)) != 0:
                return None
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:  # 1 = NVML_CLOCK_SM
                self.smax = float(mx.value)
            lim = ctypes.c_uint()
            get_lim = getattr(lib, "nvmlDeviceGetEnforcedPowerLimit", None)
            if get_lim is not None and get_lim(h, ctypes.byref(lim)) == 0:  # mW, read only
                self.power_limit_w = lim.value / 1000.0
            return (lib, h)
        except (OSError, AttributeError):
            return None

    def _nvml_loop(self):
        import ctypes
        lib, h = self.nvml
        clk = ctypes.c_uint()
        mw = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        get_power = getattr(lib, "nvmlDeviceGetPowerUsage", None)
        while not self._stop.is_set():
            if not self._on.wait(0.05):
                continue
            reg = self.by_region.setdefault(self.region, ([], []))
            if lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0:
                self.sm.append(float(clk.value))
                reg[0].append(float(clk.value))
            if get_power is not None and get_power(h, ctypes.byref(mw)) == 0:
                reg[1].append(mw.value / 1000.0)
            if lib.nvmlDeviceGetCurrentClocksThrottleReasons(h, ctypes.byref(rs)) == 0:
                for bit, name in self.REASONS.items():
                    if rs.value & bit:
                        self.reasons.add(name)
            time.sleep(0.005)

    class _Active:
        def __init__(self, outer, region):
            self.o = outer
            self.region = region

        def __enter__(self):
            self.o.region = self.region
            self.o._on.set()
            if self.o.nvml is None and self.o.proc is None:
                self.o._start_smi()

        def __exit__(self, *exc):
            self.o._on.clear()
            return False

    def active(self, region="step"):
        """Samples while the block runs; `region` names it in the per-region
        medians (SM clock and board power)."""
        return self._Active(self, region)

    def _start_smi(self):
        fields = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                  "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                  "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.pci or str(self.index), f"--query-gpu={fields}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.src = "nvidia-smi"
            self.thread = threading.Thread(target=self._smi_read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _smi_read(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.proc.stdout:
            if not self._on.is_set():
                continue
            parts = [p.strip() for p in line.strip().split(",")]
            if len(parts) < 8:
                continue
            try:
                self.sm.append(float(parts[0]))
                self.smax = max(self.smax or 0.0, float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    self.reasons.add(n)

    def stop(self):
        self._stop.set()
        self._on.clear()
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.src is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no NVML and no nvidia-smi"]}
        out = {"sm_mhz": statistics.median(self.sm) if self.sm else None,
               "sm_max_mhz": self.smax, "reasons": sorted(self.reasons), "samples": len(self.sm),
               "source": self.src}
        if self.by_region:
            out["power_limit_w"] = self.power_limit_w
            out["by_region"] = {r: {"sm_mhz": statistics.median(c) if c else None,
                                    "power_w": statistics.median(p) if p else None, "samples": len(c)}
                                for r, (c, p) in self.by_region.items()}
        return out


def pci_bus_id(dev):
    """PCI bus id of a CUDA device as NVML writes it, or None."""
    import torch
    p = torch.cuda.get_device_properties(dev)
    try:
        return f"{p.pci_domain_id:08X}:{p.pci_bus_id:02X}:{p.pci_device_id:02X}.0"
    except AttributeError:
        return None


# ------------------------------------------------------------------ our arm
def select_workload(args):
    from paper_2609_22870_gb300 import synth
    w = synth.WORKLOADS[args.workload]
    if args.gran is not None:
        import dataclasses
        w = dataclasses.replace(w, name=f"{w.name}_g{args.gran}", gran=args.gran)
    if args.tokens:
        w = synth.scaled(w, T=args.tokens, name=f"{w.name}_T{args.tokens}")
    return w


def kernels_per_step(gran, mode, T):
    """Kernel launches of one FP8 step: quantise h and W (amax + encode each
    for per-tensor scaling), the GEMM, the combine, calibration (one
    cooperative launch up to 2^18 tokens, else a pass and a decide launch per
    stage: 9 stages exact, 3 grid) and the surrogate (which takes the
    calibration's count of valid tokens, so it makes no counting pass)."""
    q = 2 if gran == 0 else 1
    calib = 1 if T <= (1 << 18) else (6 if mode == 1 else 18)
    return 2 * q + 1 + 1 + calib + 1


def run_ours(args, rank, world, local_rank):
    import torch
    from paper_2609_22870_gb300 import api, synth

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    w = select_workload(args)
    T, H, V, gran = w.T, w.H, w.V, w.gran
    h = synth.hidden_states(w, dev)
    W = synth.lm_head_weight(w, dev)
    y = synth.targets(w, dev)
    adv, mask = synth.rollout(w)
    noise = synth.old_policy_noise(w)
    # the BF16 shadow pass (Algorithm 1's reference ratios) by the library's
    # kind::f16 scorer; timed on its own below, not part of the FP8 step
    shadow_ws = torch.empty(api.bf16_token_logprobs_workspace_size(T, H, V), dtype=torch.uint8, device=dev)
    shadow = {"logp": torch.empty(T, device=dev), "lse": torch.empty(T, device=dev)}
    api.bf16_token_logprobs(h, W, y, workspace=shadow_ws, out=shadow)
    logp_bf16 = shadow["logp"].clone()
    logp_old = (logp_bf16 + noise.to(dev)).float()
    r_bf16 = torch.exp(logp_bf16 - logp_old).float()
    coef = torch.exp(logp_old).float()  # TIS weight 1 (sampler = old policy) times pi_sampler
    adv_d, mask_d = adv.to(dev), mask.to(dev)
    opts = api.calib_opts(mode=args.calib_mode)
    b = api.StepBuffers(T, H, V, gran, dev)
    stream = torch.cuda.current_stream()

    ev = [torch.cuda.Event(enable_timing=True) for _ in range(7)]

    def make_step(g, bb):
        def step(record=False):
            if record:
                ev[0].record(stream)
            api.quantize(h, g, api.ROLE_ACT, bb.h_codes, bb.h_scales, bb.q_ws)
            if record:
                ev[1].record(stream)
            api.quantize(W, g, api.ROLE_WEIGHT, bb.w_codes, bb.w_scales, bb.q_ws)
            if record:
                ev[2].record(stream)
            api.logit_partials(bb.h_codes, bb.h_scales, bb.w_codes, bb.w_scales, g, y, bb.lp_ws)
            if record:
                ev[3].record(stream)
            api.combine_logprobs(T, H, V, g, y, bb.lp_ws, logp_old, bb.logp, bb.lse, bb.ratio)
            if record:
                ev[4].record(stream)
            api.calibrate_clip_bounds(bb.ratio, r_bf16, adv_d, mask_d, coef, w.eps_low, w.eps_high, opts,
                                      bb.cal_res, bb.cal_ws)
            if record:
                ev[5].record(stream)
            api.clipped_surrogate(bb.ratio, adv_d, mask_d, None, bounds=api.bounds_view(bb.cal_res),
                                  stats=bb.stats, workspace=bb.sur_ws,
                                  out={"grad": bb.grad, "clip_mask": bb.clip_mask},
                                  n_valid=api.n_valid_view(bb.cal_res))
            if record:
                ev[6].record(stream)
        return step

    step = make_step(gran, b)

    for _ in range(args.warmup):
        step()
    api.check()
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(pci_bus_id(dev), local_rank)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    per_step_events = []
    with clocks.active():
        t0.record(stream)
        for _ in range(args.steps):
            ev[:] = [torch.cuda.Event(enable_timing=True) for _ in range(7)]
            step(record=True)
            per_step_events.append(list(ev))
        t1.record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    stage = np.zeros(6)
    for evs in per_step_events:
        stage += [evs[i].elapsed_time(evs[i + 1]) for i in range(6)]
    elapsed_ms = t0.elapsed_time(t1)
    api.check()
    # more clock samples under the same load: the step repeated (untimed)
    # for about a second with the sampler on, since the timed region itself
    # is short
    n_more = max(1, int(1000.0 / max(0.1, elapsed_ms / args.steps)))
    with clocks.active():
        for _ in range(n_more):
            step()
        torch.cuda.synchronize()

    # the same step captured once into a CUDA graph and replayed: the six
    # kernels launch from the device-side graph, not one host launch each
    # (this matters where the step is short; the results must equal the
    # eager step's bit for bit)
    graph = None
    if not args.no_graph:
        try:
            step()
            torch.cuda.synchronize()
            eager = [t.clone() for t in (b.logp, b.ratio, b.grad, b.clip_mask, b.cal_res, b.stats)]
            cg = torch.cuda.CUDAGraph()
            side = torch.cuda.Stream()
            side.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(side):
                step()
            torch.cuda.current_stream().wait_stream(side)
            with torch.cuda.graph(cg):
                step()
            cg.replay()
            torch.cuda.synchronize()
            api.check()
            same = all(torch.equal(a, c) for a, c in
                       zip(eager, (b.logp, b.ratio, b.grad, b.clip_mask, b.cal_res, b.stats)))
            for _ in range(args.warmup):
                cg.replay()
            g0 = torch.cuda.Event(enable_timing=True)
            g1 = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            g0.record()
            for _ in range(args.steps):
                cg.replay()
            g1.record()
            torch.cuda.synchronize()
            api.check()
            gms = g0.elapsed_time(g1) / args.steps
            graph = {"ms_per_step": gms, "value": whole_job_rate(T, 1, gms), "unit": "tokens/s",
                     "matches_eager": same,
                     "note": "the step captured once into a CUDA graph and replayed (torch.cuda.CUDAGraph)"}
            del cg
        except Exception as exc:  # a capture the driver refuses: report it, keep the eager figures
            graph = {"unavailable": f"{type(exc).__name__}: {str(exc)[:160]}"}

    # the same step with power-of-two block scales applied by the tensor
    # cores' block-scaled MMA (a variant outside the paper; block layout only)
    ue = None
    if gran == api.GRAN_BLOCK and not args.no_variants:
        b3 = api.StepBuffers(T, H, V, api.GRAN_BLOCK_UE8M0, dev)
        step3 = make_step(api.GRAN_BLOCK_UE8M0, b3)
        for _ in range(args.warmup):
            step3()
        torch.cuda.synchronize()
        u0 = torch.cuda.Event(enable_timing=True)
        u1 = torch.cuda.Event(enable_timing=True)
        ue_events = []
        with clocks.active("ue8m0_variant"):
            u0.record(stream)
            for _ in range(args.steps):
                ev[:] = [torch.cuda.Event(enable_timing=True) for _ in range(7)]
                step3(record=True)
                ue_events.append(list(ev))
            u1.record(stream)
            torch.cuda.synchronize()
        api.check()
        ue_stage = np.zeros(6)
        for evs in ue_events:
            ue_stage += [evs[i].elapsed_time(evs[i + 1]) for i in range(6)]
        ue_stage /= args.steps
        ue = {"ms_per_step": u0.elapsed_time(u1) / args.steps, "gemm_ms": ue_stage[2],
              "quantize_ms": ue_stage[0] + ue_stage[1]}

    # the BF16 shadow pass on its own (same inputs; the paper reruns it every
    # 20 steps, so it is reported separately and amortised)
    s0 = torch.cuda.Event(enable_timing=True)
    s1 = torch.cuda.Event(enable_timing=True)
    n_shadow = max(3, args.steps // 10)
    s0.record(stream)
    for _ in range(n_shadow):
        api.bf16_token_logprobs(h, W, y, workspace=shadow_ws, out=shadow)
    s1.record(stream)
    torch.cuda.synchronize()
    shadow_ms = s0.elapsed_time(s1) / n_shadow

    # backward through the lm_head from this step's g (dh = P W, dW = P^T h with
    # P = dLoss/dlogits recomputed from the FP8 logits), timed on its own
    bwd = ue_bwd = None
    if not args.no_backward:
        bws = torch.empty(api.lib.fp8rl_lm_head_backward_workspace_size(T, H, V), dtype=torch.uint8, device=dev)
        bout = {"dh": torch.empty(T, H, device=dev), "dW": torch.empty(V, H, device=dev)}

        def time_backward(bb, g, pow2=False):
            def backward():
                api.lm_head_backward(bb.h_codes, bb.h_scales, bb.w_codes, bb.w_scales, g, y, bb.lse, bb.grad,
                                     h, W, pow2_scales=pow2, out=bout, workspace=bws)

            backward()
            torch.cuda.synchronize()
            n_bwd = 3
            b0 = torch.cuda.Event(enable_timing=True)
            b1 = torch.cuda.Event(enable_timing=True)
            b0.record(stream)
            for _ in range(n_bwd):
                backward()
            b1.record(stream)
            torch.cuda.synchronize()
            api.check()
            return {"ms": b0.elapsed_time(b1) / n_bwd, "workspace_gb": bws.numel() / 1e9}

        bwd = time_backward(b, gran)
        if gran != api.GRAN_BLOCK_UE8M0:  # the backward's own operands on power-of-two scales
            bwd["pow2_scales"] = time_backward(b, gran, pow2=True)
        if ue is not None:  # the variant's backward: power-of-two scales throughout
            ue_bwd = time_backward(b3, api.GRAN_BLOCK_UE8M0)
        del bws, bout
    if ue is not None:
        del b3
    api.check()

    # same step through the public API with host buffers (copies inside the region)
    pin = lambda t: t.cpu().pin_memory()  # noqa: E731
    host = {"h": pin(h), "y": pin(y), "logp_old": pin(logp_old), "r_bf16": pin(r_bf16),
            "adv": pin(adv), "mask": pin(mask), "coef": pin(coef)}
    out_host = {"stats": torch.empty(b.stats.numel(), dtype=torch.uint8).pin_memory(),
                "cal": torch.empty(b.cal_res.numel(), dtype=torch.uint8).pin_memory(),
                "grad": torch.empty(T, dtype=torch.float32).pin_memory()}
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    d2h = sum(v.numel() * v.element_size() for v in out_host.values())
    # double-buffered prefetch: step i + 1's inputs are copied on a side stream
    # while step i runs (the first copy and every later one are inside the region)
    pf = api.HostBatchPrefetcher(host, dev, stream)

    def e2e_run(n):
        pf.prefetch(0, host)
        for i in range(n):
            d = pf.acquire(i % 2)
            if i + 1 < n:
                pf.prefetch((i + 1) % 2, host)
            api.score_calibrate_loss(d["h"], W, d["y"], d["logp_old"], d["r_bf16"], d["adv"], d["mask"],
                                     d["coef"], gran, w.eps_low, w.eps_high, opts, b, stream)
            pf.release(i % 2)
            out_host["stats"].copy_(b.stats, non_blocking=True)
            out_host["cal"].copy_(b.cal_res, non_blocking=True)
            out_host["grad"].copy_(b.grad, non_blocking=True)

    e2e_run(max(1, args.warmup))
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with clocks.active("e2e"):
        e0.record(stream)
        e2e_run(args.steps)
        e1.record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e2e_ms = e0.elapsed_time(e1) / args.steps
    api.check()
    clk = clocks.stop()
    fp8_cublas = measure_fp8_peak(dev) if not args.no_fp8_peak else None
    res = api.read_calib_result(b.cal_res)
    st = api.read_clip_stats(b.stats)
    # §3 diagnosis of this batch against the BF16 shadow pass (untimed)
    api.quantize(h, gran, api.ROLE_ACT, b.h_codes, b.h_scales, b.q_ws)
    api.token_logprobs(b.h_codes, b.h_scales, b.w_codes, b.w_scales, gran, y, logp_old,
                       workspace=b.lp_ws, out={"logp": b.logp, "lse": b.lse, "ratio": b.ratio})
    diag = api.read_clip_diag(api.clip_diagnostics(b.ratio, r_bf16, adv_d, mask_d, b.logp, logp_bf16,
                                                   w.eps_low, w.eps_high))
    api.check()

    ms = elapsed_ms / args.steps
    ms, e2e_ms = max_over_ranks([ms, e2e_ms], world, dev)
    if rank != 0:
        return None
    stage /= args.steps
    gemm_ms = stage[2]
    flops = 2.0 * T * H * V
    peaks, peak_src = load_peaks()
    # the timed region is well under a second at full clocks, so the burst
    # figure is the denominator; the sustained one is kept beside it
    fp8_peak = peaks["bf16_tflops"] * FP8_OVER_BF16
    fp8_peak_sus = peaks["bf16_tflops_sustained"] * FP8_OVER_BF16
    achieved = flops / (gemm_ms * 1e-3) / 1e12
    n_valid = int(mask.sum())
    line = {
        "metric": METRIC,
        "value": whole_job_rate(T, world, ms),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "fp8_e4m3 (fp32 accumulate)",
        "data": "synthetic",
        "config": {"workload": workload_desc(w), "T": T, "H": H, "V": V,
                   "granularity": GRAN_NAMES[gran],
                   "calib_mode": "grid" if args.calib_mode == 1 else "exact",
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (W codes 622 MB, bf16 W 1.2 GB); no flush",
                   "r_bf16": "from the library's BF16 shadow scorer (fp8rl_bf16_token_logprobs), "
                             "run before the timed region; timed separately under bf16_shadow"},
        "valid_tokens_per_s": whole_job_rate(n_valid, world, ms),
        "valid_tokens_per_step": n_valid,
        "roofline": {"bound": "tensor", "kernel": "fp8_gemm_kernel (logit partials)",
                     "achieved": achieved, "peak": fp8_peak, "unit": "TFLOP/s",
                     "frac": achieved / fp8_peak,
                     "peak_source": f"{peak_src} bf16 burst x {FP8_OVER_BF16:g} (nominal FP8/BF16 ratio)",
                     "achieved_def": "2*T*H*V FLOP per launch / mean CUDA-event time of the GEMM stage",
                     "peak_sustained": fp8_peak_sus, "frac_of_sustained": achieved / fp8_peak_sus,
                     "fp8_cublas_measured": fp8_cublas,
                     "traffic": measured_gemm_traffic(w), "traffic_unit": "bytes per launch"},
        "stages_ms": {"quantize_h": stage[0], "quantize_w": stage[1], "gemm_lse": stage[2],
                      "combine": stage[3], "calibrate": stage[4], "surrogate": stage[5]},
        "ms_per_step_variants": {
            "without_w_quantize": ms - stage[1],
            "calibrate_1_in_20": ms - stage[4] + stage[4] / 20,
            "note": "derived from the stage timings: W quantised once per optimiser step and shared "
                    "by both scoring passes; Algorithm 1 recalibrating every 20 steps"},
        "bf16_shadow": {"ms": shadow_ms, "tflops": flops / (shadow_ms * 1e-3) / 1e12,
                        "frac_of_bf16_peak": flops / (shadow_ms * 1e-3) / 1e12 / peaks["bf16_tflops"],
                        "frac_of_bf16_sustained": flops / (shadow_ms * 1e-3) / 1e12 / peaks["bf16_tflops_sustained"],
                        "ms_per_step_amortised_1_in_20": ms + shadow_ms / 20,
                        "note": "BF16 reference scoring of the same tokens (Algorithm 1 needs r_BF16); "
                                "the paper recomputes it every 20 steps"},
        "e2e": {"value": whole_job_rate(T, world, e2e_ms), "unit": "tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "note": "h, targets, logp_old, r_bf16, adv, mask, coef copied in from pinned host memory "
                        "(step i+1's copy overlaps step i on a side stream, double-buffered); stats, "
                        "bounds, dloss/dlogp read back every step; lm_head W is resident model state"},
        "gpu_launches": kernels_per_step(gran, args.calib_mode, T) * args.steps,
        "clocks": clk,
        "result": {"lo": res["lo_new"], "hi": res["hi_new"], "loss": st["loss"],
                   "clip_frac_pos": st["clip_frac_pos"], "clip_frac_neg": st["clip_frac_neg"]},
        "diagnostics": {k: diag[k] for k in ("over_clipped_lo", "over_clipped_hi", "clipped_lo_fp8",
                                             "clipped_hi_fp8", "clipped_lo_bf16", "clipped_hi_bf16",
                                             "nmae_prob", "nmae_ratio")},
    }
    if graph is not None:
        line["cuda_graph"] = graph
    if ue is not None:
        ue_tf = flops / (ue["gemm_ms"] * 1e-3) / 1e12
        line["ue8m0_mma_variant"] = {
            "value": whole_job_rate(T, 1, ue["ms_per_step"]), "unit": "tokens/s",
            "ms_per_step": ue["ms_per_step"], "gemm_ms": ue["gemm_ms"], "quantize_ms": ue["quantize_ms"],
            "gemm_tflops": ue_tf, "gemm_frac_of_fp8_peak": ue_tf / fp8_peak,
            "note": "the same step with power-of-two block scales (fp8rl_quantize_ue8m0, 1x128 / 128x128) "
                    "applied by tcgen05.mma kind::mxf8f6f4 with E8M0 scale factors in tensor memory; a "
                    "variant outside the paper (its scales are amax / 448), so not the headline value"}
        if ue_bwd is not None:
            ideal_ms = 3 * flops / (fp8_peak * 1e12) * 1e3
            line["ue8m0_mma_variant"]["lm_head_backward"] = {
                "ms": ue_bwd["ms"], "tflops": 3 * flops / (ue_bwd["ms"] * 1e-3) / 1e12,
                "frac_of_roofline": ideal_ms / ue_bwd["ms"],
                "note": "the variant's backward: P, P^T, W^T and h^T with power-of-two scales, the recompute "
                        "and both contractions on the block-scaled MMA"}
    if bwd is not None:
        ideal_ms = 3 * flops / (fp8_peak * 1e12) * 1e3
        bwd.update({"tflop_per_call": 3 * flops / 1e12, "tflops": 3 * flops / (bwd["ms"] * 1e-3) / 1e12,
                    "ideal_ms": ideal_ms, "frac_of_roofline": ideal_ms / bwd["ms"],
                    "note": "dh and dW from this step's dloss/dlogp: z recomputed on the FP8 GEMM whose "
                            "epilogue writes dlogits as E4M3 codes (1x128 along V, and 128x128 transposed), "
                            "W and h transposed and quantised (128x128), dh and dW on the block-scaled FP8 "
                            "GEMM; ideal = 6THV at the FP8 burst peak"})
        if "pow2_scales" in bwd:
            p2 = bwd["pow2_scales"]
            p2.update({"tflops": 3 * flops / (p2["ms"] * 1e-3) / 1e12, "frac_of_roofline": ideal_ms / p2["ms"],
                       "note": "FP8RL_BWD_POW2_SCALES: z recomputed from this step's codes as above, P, P^T, W^T "
                               "and h^T with power-of-two scales (floored at 2^-127), dh and dW on the "
                               "block-scaled MMA (kind::mxf8f6f4)"})
        line["lm_head_backward"] = bwd
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = oracle_step_estimate(w, budget_s=args.cpu_budget)
    return line


def measure_fp8_peak(dev, n=8192, burst_reps=10, sustained_s=4.0):
    """Dense E4M3 x E4M3 -> bf16 GEMM rate of the vendor library
    (torch._scaled_mm, cuBLASLt) at n^3: best of ``burst_reps`` single calls
    (burst) and the mean over back-to-back calls for ``sustained_s`` seconds
    (sustained), 2 n^3 FLOP per call.  Context for the FP8 roofline; the
    denominator stays the measured BF16 figure times the nominal ratio."""
    import torch
    try:
        g = torch.Generator(device=dev)
        g.manual_seed(1)
        a = torch.randn(n, n, device=dev, generator=g).to(torch.float8_e4m3fn)
        b = torch.randn(n, n, device=dev, generator=g).to(torch.float8_e4m3fn).t()
        one = torch.ones((), device=dev)

        def mm():
            return torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)

        for _ in range(3):
            mm()
        torch.cuda.synchronize()
        best = float("inf")
        for _ in range(burst_reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            mm()
            e1.record()
            e1.synchronize()
            best = min(best, e0.elapsed_time(e1))
        calls = 0
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t_end = time.perf_counter() + sustained_s
        e0.record()
        while time.perf_counter() < t_end:
            for _ in range(20):
                mm()
            calls += 20
            torch.cuda.current_stream().synchronize()
        e1.record()
        e1.synchronize()
        flop = 2.0 * n ** 3
        return {"burst_tflops": flop / (best * 1e-3) / 1e12,
                "sustained_tflops": flop * calls / (e0.elapsed_time(e1) * 1e-3) / 1e12,
                "how": f"torch._scaled_mm E4M3 x E4M3 -> bf16, unit scales, {n}^3; best of {burst_reps} "
                       f"(burst) and back to back for {sustained_s:g} s (sustained)"}
    except (RuntimeError, AttributeError, TypeError) as e:
        return {"unavailable": str(e).splitlines()[0][:200]}


# ------------------------------------------------------------------ oracle arm
def oracle_step_estimate(w, budget_s=20.0, seed=0):
    """Times the CPU oracle on a bounded sample of the workload and extrapolates
    to one full step: W quantisation and scoring are timed on a sample of
    128-row vocabulary strips and token rows (cost linear in both), calibration
    and the surrogate run on all T tokens (synthetic ratios of the same size)."""
    import torch
    from oracle import calibrate as OC
    from oracle import logprobs as OL
    from oracle import quantize as OQ
    from oracle import surrogate as OS
    from paper_2609_22870_gb300 import synth

    rng = np.random.default_rng(seed)
    n_rows = min(w.T, 512)
    h = synth.normal_bf16(n_rows, w.H, 1.0, 1, "cpu").float().numpy()
    t = time.perf_counter()
    hq, hs = OQ.quantize(h, w.gran, OQ.ACT)
    t_qh = (time.perf_counter() - t) / n_rows
    order = rng.permutation(w.V // 128)
    t_qw = t_gemm = 0.0
    n_strips = 0
    t_start = time.perf_counter()
    for sidx in order:  # as many strips as the time budget allows
        Wx = synth.normal_bf16(128, w.H, 0.02, int(sidx), "cpu").float().numpy()
        t = time.perf_counter()
        wq, ws = OQ.quantize(Wx, w.gran, OQ.WEIGHT)
        t_qw += time.perf_counter() - t
        t = time.perf_counter()
        z = OL.logits(hq, hs, wq, ws, w.gran)
        OL.log_softmax_gather(z, np.zeros(n_rows, np.int64))
        t_gemm += time.perf_counter() - t
        n_strips += 1
        if time.perf_counter() - t_start >= budget_s:
            break
    frac = (w.V / 128) / n_strips
    t_qw_full = t_qw * frac
    t_score_full = t_gemm * frac * (w.T / n_rows)
    adv, mask = synth.rollout(w)
    r_bf, r_fp, coef = synth.ratio_inputs(w.T, 3)
    t = time.perf_counter()
    res = OC.calibrate_clip_bounds(r_fp.numpy(), r_bf.numpy(), adv.numpy(), mask.numpy(), coef.numpy(),
                                   w.eps_low, w.eps_high)
    t_cal = time.perf_counter() - t
    t = time.perf_counter()
    OS.clipped_surrogate(r_fp.numpy(), adv.numpy(), mask.numpy(), None, res["lo_new"], res["hi_new"])
    t_loss = time.perf_counter() - t
    step_s = t_qh * w.T + t_qw_full + t_score_full + t_cal + t_loss
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {"value": w.T / step_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": (f"{n_strips}/{w.V // 128} W strips of 128 rows quantised and scored against "
                       f"{n_rows} token rows (numpy float64, BLAS threads up to {cores}); calibrate + "
                       f"surrogate on all {w.T} tokens; full step extrapolated linearly "
                       f"({step_s:.1f} s/step)"),
            "step_seconds": step_s}


def run_reference(args, rank, world):
    """The oracle arm: each step is one bounded sample of the workload (W
    strips and token rows scored, calibration and the loss on all T tokens),
    timed on the host cores.  ``ms_per_step`` is the wall time of one such
    sample; the sample stands for a fraction of a full step, so ``value``
    (tokens per second) is the full step's T over its time extrapolated from
    the sample, and ``tokens_per_step`` is the tokens that fraction is worth."""
    from paper_2609_22870_gb300 import synth
    if rank != 0:
        return None
    w = select_workload(args)
    per_step = max(0.1, 120.0 / max(1, args.steps + args.warmup))
    for i in range(args.warmup):
        oracle_step_estimate(w, budget_s=per_step, seed=100 + i)
    vals, walls = [], []
    t0 = time.perf_counter()
    for i in range(args.steps):
        t = time.perf_counter()
        vals.append(oracle_step_estimate(w, budget_s=per_step, seed=i))
        walls.append(time.perf_counter() - t)
    wall = time.perf_counter() - t0
    v = statistics.median(x["value"] for x in vals)
    full_s = statistics.median(x["step_seconds"] for x in vals)
    sample_s = statistics.median(walls)
    cb = dict(vals[0])
    cb["value"] = v
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sample_s * 1e3,
            "step_kind": "bounded sample of the workload (not a full step)",
            "tokens_per_step": v * sample_s,
            "full_step_ms_extrapolated": full_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "float64 (oracle)", "data": "synthetic",
            "config": {"workload": workload_desc(w), "T": w.T, "H": w.H, "V": w.V,
                       "granularity": GRAN_NAMES[w.gran]},
            "cpu_baseline": cb, "sample_wall_seconds": wall,
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def run_kernel_rooflines(args, local_rank):
    """HBM-bound kernels at stress sizes: bytes are the algorithmic bytes of
    one call (every input read once, every output written once), time is the
    CUDA-event average over repeated calls on inputs larger than L2.
    ``--stress-scale`` shrinks the token counts (h rows 131072, ratios 2^27)
    for profiler captures; every input stays larger than L2."""
    import torch
    from paper_2609_22870_gb300 import api, synth

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    peaks, src = load_peaks()
    hbm = peaks["hbm_gbs"]
    out = []

    def timed(fn, reps):
        fn()
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            fn()
        b.record()
        torch.cuda.synchronize()
        api.check()
        return a.elapsed_time(b) / reps

    def line(kernel, shape, nbytes, ms):
        gbs = nbytes / (ms * 1e-3) / 1e9
        out.append({"kernel": kernel, "shape": shape, "bytes": nbytes, "ms": ms, "GB/s": gbs,
                    "peak_GB/s": hbm, "frac": gbs / hbm, "peak_source": src})

    # a1/a2 quantise at the long workload's h (T 131072 x 4096) and the lm_head W
    T, H, V = max(8192, int(131072 * args.stress_scale)), 4096, 151936
    h = synth.normal_bf16(T, H, 1.0, 7, dev)
    for gran, name in ((2, "block 1x128"), (1, "row"), (0, "tensor")):
        codes = torch.empty(T, H, dtype=torch.uint8, device=dev)
        sc = torch.empty(max(1, api.scales_count(T, H, gran, 0)), dtype=torch.float32, device=dev)
        ws = torch.empty(256, dtype=torch.uint8, device=dev)
        ms = timed(lambda: api.quantize(h, gran, 0, codes, sc, ws), 10)
        line(f"quantize h ({name})", [T, H], T * H * 3 + sc.numel() * 4, ms)
    del h, codes
    W = synth.normal_bf16(V, H, 0.02, 8, dev)
    for gran, name in ((2, "block 128x128"), (1, "row")):
        codes = torch.empty(V, H, dtype=torch.uint8, device=dev)
        sc = torch.empty(max(1, api.scales_count(V, H, gran, 1)), dtype=torch.float32, device=dev)
        ms = timed(lambda: api.quantize(W, gran, 1, codes, sc), 10)
        line(f"quantize W ({name})", [V, H], V * H * 3 + sc.numel() * 4, ms)
    del W, codes

    # a4 combine at the 8B workload: 1187 (max, sum-exp) partials per token
    T = 16384
    ws = torch.empty(api.token_logprobs_workspace_size(T, H, V, 2), dtype=torch.uint8, device=dev)
    n_chunks = (V + 127) // 128
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    part = ws[: n_chunks * T * 8].view(torch.float32).view(n_chunks, T, 2)
    part[..., 0] = torch.randn(n_chunks, T, generator=g, device=dev) * 2
    part[..., 1] = torch.rand(n_chunks, T, generator=g, device=dev) * 100 + 1
    zoff = -(-(n_chunks * T * 8) // 256) * 256
    ws[zoff: zoff + T * 4].view(torch.float32).copy_(torch.randn(T, generator=g, device=dev))
    y = torch.randint(0, V, (T,), generator=g, device=dev, dtype=torch.int32)
    lp_old = torch.randn(T, generator=g, device=dev) - 11
    outs = [torch.empty(T, device=dev) for _ in range(3)]
    ms = timed(lambda: api.combine_logprobs(T, H, V, 2, y, ws, lp_old, *outs), 20)
    line("combine (logsumexp of partials)", [n_chunks, T], n_chunks * T * 8 + T * (4 + 4 + 4) + T * 12, ms)
    del ws, part

    # a5/a6 at T = 2^27 synthetic ratios
    T = max(1 << 20, int((1 << 27) * args.stress_scale))
    g = torch.Generator(device=dev)
    g.manual_seed(9)
    r_bf = torch.exp(torch.randn(T, generator=g, device=dev) * 0.05)
    r_fp = r_bf * torch.exp(torch.randn(T, generator=g, device=dev) * 0.05)
    adv = torch.randn(T, generator=g, device=dev)
    coef = torch.exp(torch.randn(T, generator=g, device=dev) * 2 - 11)
    mask = (torch.rand(T, generator=g, device=dev) < 0.9).to(torch.uint8)
    res = torch.zeros(128, dtype=torch.uint8, device=dev)
    cws = torch.empty(api.calibrate_workspace_size(T), dtype=torch.uint8, device=dev)
    for mode, name in ((0, "exact"), (1, "grid")):
        opts = api.calib_opts(mode=mode)
        ms = timed(lambda: api.calibrate_clip_bounds(r_fp, r_bf, adv, mask, coef, 0.2, 0.2, opts, res, cws), 5)
        line(f"calibrate ({name})", [T], T * 17, ms)
    grad = torch.empty(T, device=dev)
    cm = torch.empty(T, dtype=torch.uint8, device=dev)
    st = torch.zeros(128, dtype=torch.uint8, device=dev)
    sws = torch.empty(api.surrogate_workspace_size(T), dtype=torch.uint8, device=dev)
    ms = timed(lambda: api.clipped_surrogate(r_fp, adv, mask, None, 0.8, 1.2, None, stats=st, workspace=sws,
                                             out={"grad": grad, "clip_mask": cm}), 10)
    line("clipped surrogate", [T], T * (4 + 4 + 1 + 4 + 1), ms)
    n_seq = T // 512
    sid = (torch.arange(T, device=dev, dtype=torch.int64) // 512).to(torch.int32)
    qws = torch.empty(api.lib.fp8rl_surrogate_seq_mean_workspace_size(T, n_seq), dtype=torch.uint8, device=dev)
    ms = timed(lambda: api.clipped_surrogate_seq_mean(r_fp, adv, sid, n_seq, mask, None, 0.8, 1.2, stats=st,
                                                      workspace=qws, out={"grad": grad, "clip_mask": cm}), 10)
    line("clipped surrogate, sequence mean", [T], T * (5 + 4 + 4 + 4 + 1 + 4 + 1), ms)
    # sequence-level ratio clipping: logp, logp_old, ids, mask in; dloss/dlogp
    # out; one advantage, ratio and clip byte per response
    lp = torch.log(r_fp) - 3.0
    lpo = torch.log(r_bf) - 3.0
    a_seq = adv[:n_seq].contiguous()
    lws = torch.empty(api.lib.fp8rl_seq_level_surrogate_workspace_size(T, n_seq), dtype=torch.uint8, device=dev)
    s_ratio = torch.empty(n_seq, device=dev)
    s_clip = torch.empty(n_seq, dtype=torch.uint8, device=dev)
    ms = timed(lambda: api.seq_level_clipped_surrogate(lp, lpo, a_seq, sid, mask, 0.8, 1.2, stats=st,
                                                       workspace=lws, out={"grad": grad, "seq_ratio": s_ratio,
                                                                           "seq_clip": s_clip}), 10)
    line("clipped surrogate, sequence-level ratio", [T], T * (4 + 4 + 4 + 1 + 4) + n_seq * 9, ms)
    del qws, sid
    lp8 = torch.log(r_fp)
    lpb = torch.log(r_bf)
    dbuf = torch.zeros(256, dtype=torch.uint8, device=dev)
    dws = torch.empty(api.lib.fp8rl_clip_diagnostics_workspace_size(T), dtype=torch.uint8, device=dev)
    ms = timed(lambda: api.clip_diagnostics(r_fp, r_bf, adv, mask, lp8, lpb, 0.2, 0.2, out=dbuf, workspace=dws), 10)
    line("over-clip / NMAE diagnostics", [T], T * (4 * 5 + 1), ms)
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="grpo_8b")
    ap.add_argument("--gran", type=int, default=None, help="override the granularity (0 tensor, 1 row, 2 block)")
    ap.add_argument("--tokens", type=int, default=0, help="score this many tokens instead (a smaller case)")
    ap.add_argument("--calib-mode", type=int, default=0)
    ap.add_argument("--cpu-budget", type=float, default=20.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-backward", action="store_true", help="skip timing the lm_head backward")
    ap.add_argument("--no-fp8-peak", action="store_true", help="skip measuring the vendor FP8 GEMM rate")
    ap.add_argument("--no-graph", action="store_true", help="skip timing the step replayed from a CUDA graph")
    ap.add_argument("--no-variants", action="store_true",
                    help="skip timing the step with power-of-two scales on the block-scaled MMA")
    ap.add_argument("--kernels", action="store_true",
                    help="print HBM rooflines of the memory-bound kernels at stress sizes instead")
    ap.add_argument("--stress-scale", type=float, default=1.0,
                    help="--kernels: fraction of the stress token counts (for profiler captures)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.kernels:
        for item in run_kernel_rooflines(args, local_rank):
            print(json.dumps(item), flush=True)
        return
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        import torch
        if world > 1:
            import torch.distributed as dist
            torch.cuda.set_device(local_rank)
            dist.init_process_group("nccl")
        line = run_ours(args, rank, world, local_rank)
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
