"""The multi-rank host logic of bench.py on CPU: two gloo ranks on 127.0.0.1.

The path has no exchange step, so N GPUs run N replicas; the ranks meet only at the barriers
around the timed region and for the maximum of their times, and rank 0 alone runs the CPU
reference arm.  These are exercised here with world_size 2 over gloo.
"""
import argparse
import os
import socket

import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench._rank_barrier(world)
        ms = bench._max_over_ranks(10.0 + 5.0 * rank, world, "cpu")  # rank 1 is slower
        value = bench._job_throughput(world, 1000, ms)
        bench._rank_barrier(world)
        out.put((rank, ms, value, bench._dist()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_time_and_the_job_total():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    results = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, value, (r, world, local) in results:
        assert ms == 15.0                      # the maximum over ranks, on every rank
        assert value == 2 * 1000 / 0.015       # both ranks' units in the slowest rank's time
        assert (r, world, local) == (rank, 2, rank)


def test_single_rank_needs_no_process_group():
    assert bench._max_over_ranks(3.5, 1, "cpu") == 3.5
    bench._rank_barrier(1)
    assert bench._job_throughput(1, 100, 2.0) == 100 / 0.002


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    ns = argparse.Namespace(workload="llama8b_l8192", steps=1, warmup=0)
    assert bench.run_reference(ns) is None     # returns at once, prints nothing
    assert capsys.readouterr().out == ""
