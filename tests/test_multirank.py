"""Host logic of the multi-GPU bench path (replicas only, no collective on the data path),
exercised with world-size-2 gloo process groups on the CPU: each replica draws its own
sequences, the job's time is the slowest rank's and its tokens the sum over ranks, and the
reference arm runs on rank 0 only."""
import argparse
import multiprocessing as mp
import os
import socket

import pytest

import bench
import synth_inputs as S


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms, tok = bench.job_totals(10.0 + 5.0 * rank, 100 * (rank + 1), world, "cpu")
        q.put((rank, ms, tok))
    finally:
        dist.destroy_process_group()


def test_job_totals_take_max_time_and_sum_tokens_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs)
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, ms, tok in got:
        assert ms == 15.0 and tok == 300, (rank, ms, tok)


def test_job_totals_single_rank_is_identity():
    assert bench.job_totals(3.5, 7, 1, "cpu") == (3.5, 7)


def test_replicas_draw_different_sequences_from_the_same_seed():
    args = argparse.Namespace(seed=1, batch=8, ctx_lo=768, ctx_hi=1024)
    shape = S.ModelShape()
    c0, p0 = bench.sequence_inputs(args, shape, rank=0)
    c1, p1 = bench.sequence_inputs(args, shape, rank=1)
    assert (c0, p0) == bench.sequence_inputs(args, shape, rank=0)   # reproducible
    assert c0 != c1 and p0 != p1
    assert all(768 <= c <= 1024 for c in c0 + c1)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    def no_work(*a, **k):
        raise AssertionError("a non-zero rank must not build the workload")

    monkeypatch.setattr(bench, "workload", no_work)
    monkeypatch.setenv("RANK", "1")
    assert bench.run_reference(argparse.Namespace()) is None
