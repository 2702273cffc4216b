"""The benchmark's N > 1 host logic, on CPU with two gloo ranks.

The decode path runs as replicas on N GPUs (no collective on the data path): each rank times its
own token stream, the job's step time is the slowest rank's, and the whole-job rate counts every
rank's tokens.  These tests run the same helpers bench.py uses under torchrun, with the gloo
backend on 127.0.0.1, and check the reference arm's rule that only rank 0 works and prints.
"""
from __future__ import annotations

import os
import socket
import subprocess
import sys
from pathlib import Path

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = Path(__file__).resolve().parents[1]


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, values, out_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, str(ROOT))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # the repeat count and the median step time of each rank: every rank leaves with the max
        reps = int(bench.all_ranks_max(torch, values[rank][0], "cpu"))
        ms = bench.all_ranks_max(torch, values[rank][1], "cpu")
        dist.barrier()
        out_q.put((rank, reps, ms, bench.replicas_tok_s(world, ms)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_whole_job_rate_gloo():
    world, port = 2, _free_port()
    values = [(3, 2.75), (5, 2.5)]  # (timed-region repeats, ms per step) seen by ranks 0 and 1
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, values, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, reps, ms, tok_s in got:
        assert reps == 5, "every rank must time the same number of repeats (the largest)"
        assert ms == 2.75, "the job's step time is the slowest rank's"
        assert tok_s == pytest.approx(2 * 1000.0 / 2.75), "whole-job rate: both replicas' tokens"


def test_one_process_needs_no_group():
    sys.path.insert(0, str(ROOT))
    import bench
    assert not dist.is_initialized()
    assert bench.all_ranks_max(torch, 4.5, "cpu") == 4.5
    assert bench.replicas_tok_s(1, 2.5) == pytest.approx(400.0)


def test_reference_arm_runs_on_rank_zero_only():
    """Under torchrun the reference arm's other ranks exit 0 at once, without work or output."""
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1",
               MASTER_PORT=str(_free_port()))
    r = subprocess.run([sys.executable, str(ROOT / "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "2",
                        "--warmup", "3"], capture_output=True, text=True, timeout=300, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""
