"""The multi-process host logic of the benchmark on CPU (gloo, world size 2).

The GPU path shards by sequence with no data exchange (replicas, weak
scaling); what ranks share is the timing: a barrier, the slowest rank's time
as the job's time, and the whole-job rate over all ranks. The reference arm
runs on rank 0 alone.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, local = bench.rank_env()
        assert (w, r, local) == (world, rank, rank)
        dist.barrier()
        ms = bench.max_over_ranks(100.0 + 25.0 * rank, world, "cpu")
        rate = bench.whole_job_rate(16 * 256, world, ms)
        # each rank draws its own batch from a rank-dependent seed
        k, _ = synth.make_kv(bench.layer_seed(0) + 100000 * rank, 1, 1, 8)
        digest = float(np.abs(k).sum())
        got = [None] * world
        dist.all_gather_object(got, (ms, rate, digest))
        out[rank] = got
    finally:
        dist.destroy_process_group()


def test_two_ranks_time_by_the_slowest_and_sum_units():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(world):
        ranks = out[r]
        assert [x[0] for x in ranks] == [125.0, 125.0]          # max over ranks, on every rank
        assert ranks[0][1] == pytest.approx(16 * 256 * 2 / 0.125)
        assert ranks[0][2] != ranks[1][2]                         # different inputs per rank


def test_single_process_helpers_are_identity():
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
    assert bench.whole_job_rate(4096, 1, 1000.0) == 4096.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    called = []
    monkeypatch.setattr(bench, "oracle_sample", lambda *a, **k: called.append(1))
    args = type("A", (), {"steps": 1, "warmup": 1, "ref_decode_steps": 1})()
    assert bench.run_reference(args, synth.workload("long_context_32k")) is None
    assert called == [] and capsys.readouterr().out == ""
