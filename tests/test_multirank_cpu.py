"""The bench's multi-rank path on CPU: two gloo ranks, no GPU.

Under torchrun every rank runs its own batch (weak scaling) with no
collective on the data path; the only exchange is the max over ranks of the
timed region, from which rank 0 reports the whole-job throughput.
"""
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, ms_of_rank, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_00531_gb300 import workload as W
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(ms_of_rank[rank], world, torch.device("cpu"))
        w = W.WORKLOADS["tiny"]
        d = W.draft_block(w, seed=bench.rank_seed(w.seed, rank))
        digest = float(np.asarray(W.bf16_to_f64(d.logits)).sum())
        q.put((rank, ms, bench.job_steps_per_s(ms, 20, world), digest))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_draw_their_own_batches():
    world, port = 2, _free_port()
    ms_of_rank = [10.0, 15.5]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, ms_of_rank, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    for p in procs:
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    # every rank sees the slowest rank's time
    assert [g[1] for g in got] == [15.5, 15.5]
    # whole-job throughput: steps of all ranks over that time
    assert got[0][2] == pytest.approx(2 * 20 / 0.0155)
    assert got[0][2] == got[1][2]
    # weak scaling: each rank draws a different batch of the same shape
    assert got[0][3] != got[1][3]


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.25, 1, torch.device("cpu")) == 3.25
    assert bench.job_steps_per_s(1000.0, 20, 1) == pytest.approx(20.0)
    assert bench.rank_seed(5, 0) == 5 and bench.rank_seed(5, 1) != 5


def test_reference_arm_prints_only_on_rank_zero(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.main()
    assert buf.getvalue() == ""
