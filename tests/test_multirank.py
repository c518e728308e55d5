"""The multi-GPU path of bench.py is replicas only (utterances are independent,
the verify step has no exchange): each rank decodes its own batch, and the job
is timed by the slowest rank.  These are the host-side pieces of that path,
run as two gloo ranks on the CPU."""
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


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        my_seconds = [1.5, 2.5][rank]
        slowest = bench.max_over_ranks(dist, my_seconds, device="cpu")
        rate = bench.whole_job_rate(world, 3, 100, slowest)
        dist.barrier()
        q.put((rank, slowest, rate))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(world))
    for rank, slowest, rate in got:
        assert slowest == 2.5                       # max over ranks, on every rank
        assert rate == pytest.approx(2 * 3 * 100 / 2.5)   # all ranks' tokens over the slowest time


def test_single_process_needs_no_group():
    assert bench.max_over_ranks(None, 1.25) == 1.25
    assert bench.whole_job_rate(1, 2, 50, 0.5) == 200.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    args = type("A", (), {"config": "tiny-fp32-b1-k4", "steps": 1, "warmup": 3})()
    assert bench.run_reference(args) is None
    assert capsys.readouterr().out == ""
