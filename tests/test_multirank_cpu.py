"""The N > 1 bench path on CPU: two gloo ranks (127.0.0.1) run the replica
timing reduction bench.py uses over NCCL on GPUs, and a non-zero rank
of the reference arm exits without work or output.

The path itself has no data-path collective (each GPU scores its own replica
of the workload); the only exchange is the max over ranks of the timings.
"""

import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms, e2e = bench.max_over_ranks([10.0 + rank, 20.0 - 3 * rank], world, "cpu")
        q.put((rank, ms, e2e, bench.whole_job_rate(16384, world, ms)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_max_and_scale_weakly():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for rank, ms, e2e, rate in got:
        assert ms == 11.0 and e2e == 20.0  # slowest rank of each figure
        assert rate == pytest.approx(2 * 16384 / 11e-3)


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([3.5, 7.0], 1) == [3.5, 7.0]
    assert bench.whole_job_rate(100, 1, 10.0) == pytest.approx(1e4)


def test_reference_arm_nonzero_rank_exits_quietly():
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0
    assert r.stdout.strip() == ""
