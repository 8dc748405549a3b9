"""The bench's multi-rank path on CPU (gloo, world size 2).

The path has no cross-rank exchange: every rank runs its own replica on its
own layer (weak scaling), the ranks meet at barriers around the timed region,
the job's time is the slowest rank's (a MAX all-reduce), and rank 0 alone
prints. These tests run that host logic in two spawned processes.
"""
import os
import socket

import numpy as np
import pytest

import bench
from paper_2512_21859_gb300 import inputs


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _timing_worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    w, r, _ = bench.dist_env()
    dist = bench.dist_init(w, use_cuda=False)
    try:
        dist.barrier()
        slowest = bench.max_over_ranks(dist, 10.0 + 5.0 * r)  # rank 1 took longer
        dist.barrier()
        q.put((r, w, slowest))
    finally:
        dist.destroy_process_group()


def test_job_time_is_the_slowest_rank_over_gloo():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_timing_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(q.get(timeout=10) for _ in range(2))
    assert got == [(0, 2, 15.0), (1, 2, 15.0)]


def test_single_rank_needs_no_process_group():
    assert bench.dist_init(1, use_cuda=False) is None
    assert bench.max_over_ranks(None, 3.5) == 3.5


def test_job_value_is_the_sum_over_replicas():
    one = bench.job_value(1, 376.3e6, 30, 5.0)
    assert one == pytest.approx(376.3e6 * 30 / 5e-3 / 1e9)
    assert bench.job_value(2, 376.3e6, 30, 5.0) == pytest.approx(2 * one)


def test_replicas_get_independent_layers():
    wl = inputs.WORKLOADS["tiny"]
    a0, a1 = inputs.make_layer(wl, 0), inputs.make_layer(wl, 1)
    assert not np.array_equal(a0["K"], a1["K"])  # rank-seeded: each rank its own layer
    assert np.array_equal(a0["K"], inputs.make_layer(wl, 0)["K"])  # and reproducible


def test_reference_arm_prints_on_rank_zero_only(monkeypatch, capsys):
    argv = ["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "0"]
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    assert bench.main(argv) == 0
    assert capsys.readouterr().out == ""
    monkeypatch.setenv("RANK", "0")
    assert bench.main(argv) == 0
    out = capsys.readouterr().out.strip().splitlines()
    assert len(out) == 1 and '"impl": "reference"' in out[0]
