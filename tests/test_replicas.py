"""The multi-GPU path is replicas only: each rank runs its own workload and
rank 0 reports the whole job (all ranks' bytes over the slowest rank's time).
Its host logic runs here as two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import workloads as W


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # rank r pretends its timed region took (r + 1) ms and e2e 10 (r + 1) ms
        got = bench.max_over_ranks([rank + 1.0, 10.0 * (rank + 1)], "cpu", world)
        batch = bench.make_batch("tiny", "cpu", rank)
        import argparse
        args = argparse.Namespace(workload="tiny", steps=1, warmup=0)
        ref = bench.run_reference(args, rank, world) if rank != 0 else "rank0"
        q.put((rank, got, int(batch.seq_lens.sum()), float(batch.layers[0].q.float().sum()), ref))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_report_the_slowest_rank_and_distinct_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict((r[0], r[1:]) for r in (q.get(timeout=120) for _ in procs))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert res[0][0] == res[1][0] == [2.0, 20.0]  # the max of each timing over both ranks
    assert res[0][2] != res[1][2]                  # each replica draws its own inputs
    assert res[1][3] is None                       # only rank 0 runs the reference arm


def test_whole_job_value_counts_every_rank():
    assert bench.whole_job_gbs(10**9, 1, 1000.0) == pytest.approx(1.0)
    assert bench.whole_job_gbs(10**9, 4, 1000.0) == pytest.approx(4.0)
    assert bench.max_over_ranks([3.0, 4.0], "cpu", 1) == [3.0, 4.0]


def test_default_run_covers_every_configuration():
    # one default bench run times the mixed headline and, under "configs",
    # the other four configurations of the workload recipe
    names = {n for n, _ in bench.OTHER_CONFIGS}
    assert names | {"mixed"} == {"tiny", "decode", "mixed", "long", "rollout"}
    assert names <= set(W.CONFIGS)
    assert all(steps >= 8 for _, steps in bench.OTHER_CONFIGS)
