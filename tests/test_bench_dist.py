"""CPU tests of bench.py's multi-process logic (gloo, world size 2): the
timing aggregation is a max over ranks, every rank's work counts in the
whole-job value (replicas, weak scaling), and the reference arm runs on rank
0 only.  No GPU and no data-path collective are involved."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      BENCH_DIST_BACKEND="gloo")
    d, r, w = bench.dist_setup()
    assert (r, w) == (rank, world)
    local_ms = 1.0 + 0.5 * rank
    bench.barrier(d)
    worst = bench.max_over_ranks(d, local_ms)
    q.put((rank, worst))
    d.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = dict(q.get(timeout=10) for _ in range(2))
    assert got == {0: 1.5, 1: 1.5}


def test_single_process_needs_no_process_group(monkeypatch):
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    assert bench.dist_setup() == (None, 0, 1)
    assert bench.max_over_ranks(None, 3.25) == 3.25


def test_reference_arm_runs_on_rank0_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    args = type("A", (), {"warmup": 1, "steps": 1, "gpus": 2})()
    assert bench.run_reference(args, bench.workloads.llama_layer_T2048()) == 0
    assert capsys.readouterr().out == ""
