"""The N-rank path of bench.py on CPU: two ranks as processes over gloo.

Each rank runs its own robots (replicas, weak scaling; the step itself has
no exchange between ranks), so what N > 1 adds on the host is: the job is as
slow as its slowest rank (max over ranks of the timed region and of the
end-to-end time), the whole-job rate counts every rank's robots, every rank
draws its own robots' seeds, and the reference arm runs on rank 0 only.
"""
import io
import os
import socket
from contextlib import redirect_stdout

import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import argparse

        import bench
        import synth
        slowest = bench.max_over_ranks(10.0 + rank, world, device="cpu")
        fastest = -bench.max_over_ranks(-(10.0 + rank), world, device="cpu")
        seeds = synth.robot_seeds(7 + 1000 * rank, 4)
        out = io.StringIO()
        args = argparse.Namespace(gpus=world, steps=1, warmup=0)
        with redirect_stdout(out):
            if rank != 0:   # rank 0 would time the oracle; the others must return at once
                bench.run_reference(args, synth.PRESETS["tiny_fp32_b1"], rank)
        q.put((rank, slowest, fastest, seeds.tolist(), out.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_ranks_agree_on_the_slowest_time_and_run_their_own_robots():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, slow0, fast0, seeds0, out0), (r1, slow1, fast1, seeds1, out1) = res
    assert (r0, r1) == (0, 1)
    assert slow0 == slow1 == 11.0 and fast0 == fast1 == 10.0
    assert not set(seeds0) & set(seeds1)          # replicas run different robots
    assert out1 == ""                              # the reference arm prints on rank 0 only


def test_whole_job_rate_counts_every_rank():
    import bench
    assert bench.whole_job_rate(1, 64, 30, 0.15) == pytest.approx(64 * 30 / 0.15)
    assert bench.whole_job_rate(4, 64, 30, 0.15) == pytest.approx(4 * 64 * 30 / 0.15)
    assert bench.max_over_ranks(3.5, 1) == 3.5     # single rank: no collective
    assert np.isfinite(bench.whole_job_rate(8, 1, 1, 1e-3))
