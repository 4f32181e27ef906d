"""Seeded synthetic workloads shaped like the paper's 8B-32B GRPO/DAPO batches.

This module only draws random numbers and lays them out; it holds none of the
scoring, quantisation, calibration or loss arithmetic.  Both the CUDA path and
the CPU oracle take their inputs from here.

The paper trains Qwen3-8B/14B and Qwen2.5-32B with GRPO (8 responses per
prompt, §5.1 and the experiment settings of the appendix) and DAPO (16
responses per prompt, §5.2) at 16K-20K context.  Its datasets and weights are
not available, so synthetic tensors stand in for them:

* hidden states h ~ N(0, 1) and lm_head weights W ~ N(0, 0.02^2), rounded to
  bf16 (round to nearest even);
* sampled token ids y ~ U[0, V);
* one Bernoulli(p) reward per response; GRPO group-normalised advantages
  A_i = (R_i - mean(R)) / (std(R) + 1e-6) with the unbiased sample std,
  broadcast to the response's tokens (an all-equal group gets A = 0);
* a response-length mask (lengths ~ U[lo, hi]) where the workload has one,
  and the DAPO dynamic-sampling filter (groups whose rewards are all equal get
  mask 0) where the workload asks for it.

Ratio-level inputs for the calibration and loss stages (used where the FP8
scorer is not run) are drawn as log-normal perturbations around 1, see
``ratio_inputs``.
"""

import dataclasses

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    T: int               # scored tokens (rows)
    H: int               # hidden size
    V: int               # vocabulary size
    gran: int            # 0 tensor, 1 row, 2 block
    prompts: int
    group: int           # responses per prompt (G)
    resp_len: int        # tokens per response slot
    reward_p: float
    eps_low: float
    eps_high: float
    length_mask: tuple = None      # (lo, hi) response lengths, or None
    filter_equal_groups: bool = False
    seed: int = 0


GRAN_TENSOR, GRAN_ROWWISE, GRAN_BLOCK = 0, 1, 2

WORKLOADS = {
    # 1 prompt x 4 responses x 512 tokens, hidden 512, vocab 4096, per-tensor.
    "tiny_grpo": Workload("tiny_grpo", 2048, 512, 4096, GRAN_TENSOR, 1, 4, 512,
                          0.5, 0.2, 0.2, None, False, 1001),
    # 4 prompts x 8 responses x 512, Qwen3-8B lm_head (4096 x 151936), block.
    "grpo_8b": Workload("grpo_8b", 16384, 4096, 151936, GRAN_BLOCK, 4, 8, 512,
                        0.5, 0.2, 0.2, (64, 512), False, 1002),
    # 4 prompts x 16 responses x 512, Qwen2.5-32B lm_head (5120 x 151936), DAPO.
    "dapo_32b": Workload("dapo_32b", 32768, 5120, 151936, GRAN_BLOCK, 4, 16, 512,
                         0.3, 0.2, 0.28, None, True, 1003),
    # 1 prompt x 8 responses x 16384 tokens, 8B lm_head, block.
    "long_8b": Workload("long_8b", 131072, 4096, 151936, GRAN_BLOCK, 1, 8, 16384,
                        0.5, 0.2, 0.2, None, False, 1005),
}


def granularity_sweep(gran):
    """The 8B GRPO workload with the same seed at another granularity."""
    w = WORKLOADS["grpo_8b"]
    return dataclasses.replace(w, name=f"grpo_8b_g{gran}", gran=gran)


def scaled(w, T=None, H=None, V=None, name=None):
    """A smaller copy of a workload (same recipe) for tests the oracle can finish."""
    T = w.T if T is None else T
    group = w.group
    prompts = max(1, T // (group * w.resp_len)) if T >= group * w.resp_len else 1
    resp_len = max(1, T // (prompts * group))
    lm = w.length_mask
    if lm is not None:
        lm = (min(lm[0], resp_len), resp_len)
    return dataclasses.replace(w, name=name or f"{w.name}_small", T=T,
                               H=w.H if H is None else H, V=w.V if V is None else V,
                               prompts=prompts, resp_len=resp_len, length_mask=lm)


def _gen(seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def normal_bf16(rows, cols, std, seed, device="cpu", chunk_rows=8192):
    """N(0, std^2) rounded to bf16, drawn in row chunks to bound scratch memory."""
    out = torch.empty(rows, cols, dtype=torch.bfloat16, device=device)
    g = _gen(seed, device)
    for r0 in range(0, rows, chunk_rows):
        r1 = min(rows, r0 + chunk_rows)
        x = torch.randn(r1 - r0, cols, generator=g, device=device, dtype=torch.float32)
        if std != 1.0:
            x.mul_(std)
        out[r0:r1] = x.to(torch.bfloat16)
    return out


def hidden_states(w, device="cpu"):
    return normal_bf16(w.T, w.H, 1.0, w.seed * 10 + 1, device)


def lm_head_weight(w, device="cpu"):
    return normal_bf16(w.V, w.H, 0.02, w.seed * 10 + 2, device)


def targets(w, device="cpu"):
    g = _gen(w.seed * 10 + 3, "cpu")
    return torch.randint(0, w.V, (w.T,), generator=g, dtype=torch.int64).to(torch.int32).to(device)


def rollout(w, force_equal_prompt=None):
    """(adv float32 [T], mask uint8 [T]) for the workload's group layout (CPU).

    ``force_equal_prompt``: index of a prompt whose responses all get reward 1
    (an all-equal group, for tests of the DAPO dynamic-sampling filter)."""
    g = _gen(w.seed * 10 + 4, "cpu")
    n_resp = w.prompts * w.group
    R = (torch.rand(w.prompts, w.group, generator=g, dtype=torch.float64) < w.reward_p).double()
    if force_equal_prompt is not None:
        R[force_equal_prompt] = 1.0
    mean = R.mean(dim=1, keepdim=True)
    std = R.std(dim=1, keepdim=True) if w.group > 1 else torch.zeros_like(mean)
    A = ((R - mean) / (std + 1e-6)).float().reshape(n_resp)
    slot = torch.arange(w.resp_len)
    if w.length_mask is not None:
        lo, hi = w.length_mask
        lengths = torch.randint(lo, hi + 1, (n_resp,), generator=g)
        m = (slot[None, :] < lengths[:, None])
    else:
        m = torch.ones(n_resp, w.resp_len, dtype=torch.bool)
    if w.filter_equal_groups:
        equal = (R.max(dim=1).values == R.min(dim=1).values)       # [prompts]
        keep = (~equal).repeat_interleave(w.group)                 # [n_resp]
        m = m & keep[:, None]
    adv = A[:, None].expand(n_resp, w.resp_len).reshape(-1)
    mask = m.reshape(-1).to(torch.uint8)
    T = w.T
    if adv.numel() < T:  # pad the tail (T not a multiple of the layout) as invalid
        pad = T - adv.numel()
        adv = torch.cat([adv, torch.zeros(pad)])
        mask = torch.cat([mask, torch.zeros(pad, dtype=torch.uint8)])
    return adv[:T].contiguous(), mask[:T].contiguous()


def old_policy_noise(w, std=0.05):
    """N(0, std^2) per token: logp_old = logp_bf16 + noise (so r_bf16 = exp(-noise))."""
    g = _gen(w.seed * 10 + 5, "cpu")
    return (torch.randn(w.T, generator=g, dtype=torch.float64) * std).float()


def ratio_inputs(T, seed, sigma_old=0.05, sigma_fp8=0.05, logp_mean=-11.0,
                 logp_std=2.0, tie_every=0):
    """Synthetic (r_bf16, r_fp8, coef) with the statistics of the scored path.

    log r_bf16 ~ N(0, sigma_old^2) (old-policy drift), log r_fp8 = log r_bf16 +
    N(0, sigma_fp8^2) (FP8 scoring noise), coef = pi_sampler = exp(logp_old) with
    logp_old ~ N(logp_mean, logp_std^2).  ``tie_every`` > 0 copies values so
    that ratios repeat (tests of tie handling).  Returned as float32 on the CPU.
    """
    g = _gen(seed, "cpu")
    d_old = torch.randn(T, generator=g, dtype=torch.float64) * sigma_old
    d_fp8 = torch.randn(T, generator=g, dtype=torch.float64) * sigma_fp8
    lp = torch.randn(T, generator=g, dtype=torch.float64) * logp_std + logp_mean
    r_bf16 = torch.exp(d_old).float()
    r_fp8 = torch.exp(d_old + d_fp8).float()
    coef = torch.exp(lp).float()
    if tie_every:
        idx = torch.arange(T) // tie_every * tie_every
        r_fp8 = r_fp8[idx].contiguous()
        r_bf16 = r_bf16[idx].contiguous()
    return r_bf16, r_fp8, coef
