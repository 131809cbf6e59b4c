"""The benchmark's multi-rank logic on CPU: two gloo ranks on 127.0.0.1.

Every rank processes its own batch (rows are independent), so the only
exchanges are a barrier and the maximum over ranks of the timed region.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        got = bench.max_over_ranks(10.0 + 5.0 * rank, world)
        # the reference arm runs on rank 0 only; other ranks return at once
        class A:  # minimal argument object
            workload, mode, steps, warmup = 3, "cis", 1, 0
        other = bench.run_reference(A, rank, world) if rank != 0 else None
        q.put((rank, got, other))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_rank_gating_with_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [15.0, 15.0]
    assert res[1][2] is None
