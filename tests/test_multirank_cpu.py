"""World-size-2 runs of bench.py's replica plumbing on CPU (gloo).

The multi-GPU path is replicas only: every rank runs its own streams with
no collective on the data path; ranks meet at barriers and take the slowest
rank's time, and the value counts the stream-frames of all ranks.  These
tests run that plumbing with two gloo ranks, and check that a non-zero rank
of the reference arm exits without output and that ranks draw different
streams.
"""
from __future__ import annotations

import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    ranks = bench.Ranks(backend="gloo", device="cpu")
    ranks.barrier()
    slowest = ranks.max(10.0 + 2.0 * rank)          # ms; rank 1 is the slower one
    value = bench.replica_value(ranks.world, 30, slowest)
    ranks.barrier()
    q.put((rank, ranks.world, slowest, value))
    ranks.close()


def test_two_gloo_ranks_take_the_slowest_time_and_count_all_frames():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    sys.path.insert(0, ROOT)
    import bench
    for rank, world, slowest, value in got:
        assert world == 2
        assert slowest == 12.0
        assert value == pytest.approx(2 * bench.N_STREAMS * 30 / 0.012)


def test_reference_arm_nonzero_rank_exits_quietly():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    p = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0"], cwd=ROOT,
                       env=env, capture_output=True, text=True, timeout=120)
    assert p.returncode == 0
    assert p.stdout.strip() == ""


def test_ranks_draw_different_streams():
    """Rank r's replica uses streams r*8 .. r*8+7 of the generator."""
    sys.path.insert(0, ROOT)
    import synth
    a = synth.make_workload("c4", density=0.1, T=2, n=1, h=16, w=16, c=8, block=8, stream_offset=0)
    b = synth.make_workload("c4", density=0.1, T=2, n=1, h=16, w=16, c=8, block=8, stream_offset=8)
    fa = [np.array(f) for _, f in a.frames]
    fb = [np.array(f) for _, f in b.frames]
    assert not np.array_equal(fa[0], fb[0])
