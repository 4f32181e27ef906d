"""GPU: the whole step captured into a CUDA graph and replayed.

Every call of the path runs on the stream it is given, with caller-owned
buffers and workspaces and no host synchronisation, so the six launches of a
step (quantise h and W, the FP8 GEMM, the combine, the cooperative
calibration, the surrogate) can be captured once and replayed.  The replay
must reproduce the eager step's outputs bit for bit, and pick up new inputs
written into the captured tensors.
"""

import pytest
import torch

from paper_2609_22870_gb300 import synth

pytestmark = pytest.mark.gpu


def _inputs(T, H, V, seed):
    h = synth.normal_bf16(T, H, 1.0, seed, "cuda")
    W = synth.normal_bf16(V, H, 0.02, seed + 1, "cuda")
    g = torch.Generator().manual_seed(seed + 2)
    y = torch.randint(0, V, (T,), generator=g).to(torch.int32).cuda()
    logp_old = (torch.randn(T, generator=g) * 0.05 - 8.0).float().cuda()
    r_bf16 = torch.exp(torch.randn(T, generator=g) * 0.05).float().cuda()
    adv = torch.randn(T, generator=g).float().cuda()
    mask = (torch.rand(T, generator=g) < 0.8).to(torch.uint8).cuda()
    coef = torch.exp(torch.randn(T, generator=g) * 2 - 11).float().cuda()
    return h, W, y, logp_old, r_bf16, adv, mask, coef


def _outputs(b):
    return (b.logp, b.lse, b.ratio, b.grad, b.clip_mask, b.cal_res, b.stats)


@pytest.mark.parametrize("gran,T,H,V", [(0, 2048, 512, 4096), (2, 1024, 256, 3000), (3, 1024, 256, 3000)])
def test_step_replayed_from_a_cuda_graph_matches_eager(cuda_lib, gran, T, H, V):
    api = cuda_lib
    h, W, y, logp_old, r_bf16, adv, mask, coef = _inputs(T, H, V, 61 + gran)
    b = api.StepBuffers(T, H, V, gran, torch.device("cuda"))

    def step():
        api.score_calibrate_loss(h, W, y, logp_old, r_bf16, adv, mask, coef, gran, 0.2, 0.2, buffers=b)

    step()
    torch.cuda.synchronize()
    api.check()
    eager = [t.clone() for t in _outputs(b)]
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()
    torch.cuda.current_stream().wait_stream(side)
    with torch.cuda.graph(graph):
        step()
    for t in (b.logp, b.ratio, b.grad):
        t.fill_(float("nan"))
    graph.replay()
    torch.cuda.synchronize()
    api.check()
    for want, got in zip(eager, _outputs(b)):
        assert torch.equal(want, got)
    # new inputs written into the captured tensors: the replay follows them
    h2, _, y2, logp2, rb2, adv2, mask2, coef2 = _inputs(T, H, V, 90 + gran)
    for dst, src in ((h, h2), (y, y2), (logp_old, logp2), (r_bf16, rb2), (adv, adv2), (mask, mask2), (coef, coef2)):
        dst.copy_(src)
    graph.replay()
    torch.cuda.synchronize()
    api.check()
    replayed = [t.clone() for t in _outputs(b)]
    step()
    torch.cuda.synchronize()
    api.check()
    for want, got in zip(_outputs(b), replayed):
        assert torch.equal(want, got)
    assert not torch.equal(replayed[0], eager[0])
