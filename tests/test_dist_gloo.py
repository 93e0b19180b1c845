"""The multi-rank path of bench.py on CPU: two gloo ranks (world size 2).

A decode batch's sequences are independent problems, so under torchrun every
rank decodes its own batch (weak scaling) and the ranks exchange nothing on
the data path; the only collectives are the timing barrier and the maximum
of the per-rank step times.  These tests run that glue with gloo on the
host: no GPU is involved.
"""
from __future__ import annotations

import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench.barrier(world)
        # per-rank step times: the job is as slow as its slowest rank
        ms = bench.allreduce_max(1.5 + rank, world, torch.device("cpu"))
        bench.barrier(world)
        seed = bench.rank_seed(3, rank)
        ref = bench.run_reference(type("A", (), {"seed": 3})(), rank, world) \
            if rank != 0 else "rank0"
        q.put((rank, ms, seed, ref))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_barrier_max_and_independent_batches():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ms0, s0, ref0), (r1, ms1, s1, ref1) = res
    assert (r0, r1) == (0, 1)
    assert ms0 == ms1 == 2.5          # max over ranks, seen by both
    assert s0 != s1                   # each rank decodes its own batch
    assert ref1 is None               # the reference arm runs on rank 0 only


def test_job_value_counts_all_ranks():
    sys.path.insert(0, ROOT)
    import bench
    one = bench.job_value(1e8, 0.05, 1)
    assert bench.job_value(1e8, 0.05, 4) == pytest.approx(4 * one)
    assert one == pytest.approx(2000.0)  # 100 MB in 50 us = 2000 GB/s
