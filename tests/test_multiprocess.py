"""The multi-GPU bench path (independent replicas) on CPU: two gloo ranks
exercise the barrier, the max-over-ranks timing reduction and the whole-job
aggregation that bench.py uses under torchrun."""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench.barrier(world)
        slowest = bench.allreduce_max(10.0 + 3.0 * rank, world)
        rate = bench.whole_job_throughput(1e12, slowest, world)
        from paper_2605_30351_gb300 import synth
        w = synth.workload("tiny")
        # replicas draw distinct inputs (seeds depend on the rank)
        x = synth.draw_tokens(w, 4, 1000 + 101 * rank)
        q.put((rank, slowest, rate, float(x.float().sum())))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_reduce_max_and_aggregate():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    assert [o[1] for o in out] == [13.0, 13.0]            # both ranks see the slowest time
    assert out[0][2] == pytest.approx(2 * 1e12 / 13e-3 / 1e12)
    assert out[0][3] != out[1][3]                         # distinct replica inputs
