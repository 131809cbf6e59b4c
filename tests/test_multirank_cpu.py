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


def test_split_at_responses_balances_and_cuts_at_boundaries():
    from paper_2609_32444_gb300 import shard
    cu = [0, 100, 130, 400, 420, 600, 1000]
    for world in (1, 2, 3, 4, 8):
        sh = shard.split_at_responses(cu, world, T=1024)
        assert len(sh) == world
        assert sh[0][0] == 0 and sh[0][2] == 0
        assert sh[-1][1] == 1024 and sh[-1][3] == len(cu) - 1
        for (a0, a1, ai0, ai1), (b0, b1, bi0, bi1) in zip(sh, sh[1:]):
            assert a1 == b0 and ai1 == bi0  # contiguous rows and responses
            assert a1 in cu                 # cut at a response boundary
    # two ranks: the boundary closest to half of the 1000 tokens
    assert shard.split_at_responses(cu, 2)[0] == (0, 420, 0, 4)
    assert shard.shard_cu_seqlens(cu, 420, 4, 6) == [0, 180, 580]


def _shard_worker(rank, world, port, q):
    """One rank of a token-sharded batch, with the oracle as the per-rank
    pass: the ranks all-reduce their {N, G} and their losses over gloo."""
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import numpy as np
    import torch
    import torch.distributed as dist

    import oracle
    from paper_2609_32444_gb300 import shard, synth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        b = synth.make_batch(1)
        mask = b.mask.clone()
        mask[::7] = 0
        mask[128:192] = 0  # one response with no valid token
        cu = b.cu_seqlens.tolist()
        res = {}
        for agg in (oracle.AGG_TOKEN_MEAN, oracle.AGG_SEQ_MEAN):
            t0, t1, i0, i1 = shard.split_at_responses(cu, world, T=b.T)[rank]
            cu_l = np.array(shard.shard_cu_seqlens(cu, t0, i0, i1), np.int32)
            m_l = mask[t0:t1].numpy()
            n_l = int(m_l.sum())
            g_l = sum(1 for a, c in zip(cu_l, cu_l[1:]) if m_l[a:c].sum() > 0)
            cnt = torch.tensor([n_l, g_l], dtype=torch.int64)
            dist.all_reduce(cnt)
            P = oracle.params(lam=b.lam, agg=agg, n_global=int(cnt[0]), g_global=int(cnt[1]))
            out = oracle.loss_fwd_bwd(b.logits[t0:t1].numpy(), b.ids[t0:t1].numpy(),
                                      b.lp_infer[t0:t1].numpy(), b.adv[t0:t1].numpy(), P,
                                      mask=m_l, cu_seqlens=cu_l)
            loss = torch.tensor([out["loss"]], dtype=torch.float64)
            dist.all_reduce(loss)
            full = oracle.loss_fwd_bwd(b.logits.numpy(), b.ids.numpy(), b.lp_infer.numpy(),
                                       b.adv.numpy(), oracle.params(lam=b.lam, agg=agg),
                                       mask=mask.numpy(), cu_seqlens=np.array(cu, np.int32))
            scale = np.abs(full["terms"]).sum()
            res[agg] = dict(counts=cnt.tolist(), loss_err=abs(loss.item() - full["loss"]) / scale,
                            dz_equal=bool(np.array_equal(out["dz"], full["dz"][t0:t1])),
                            s_equal=bool(np.array_equal(out["c"], full["c"][t0:t1])))
        q.put((rank, res))
    finally:
        dist.destroy_process_group()


def test_token_sharded_pass_reproduces_the_batch_with_gloo():
    """Two gloo ranks split a batch at a response boundary, all-reduce
    {valid tokens, responses with a valid token} and their fp64 losses: the
    summed loss is the batch's (to rounding) and each rank's dlogits and
    per-token coefficients equal the batch's rows exactly, for the token-mean
    (Algorithm 1) and the sequence-mean (Eq. 1) normalisers."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, r in res:
        for agg, v in r.items():
            # 256 tokens, every 7th masked and one response of 64 masked
            n_expect = sum(1 for t in range(256) if t % 7 != 0 and not 128 <= t < 192)
            assert v["counts"][0] == n_expect
            if agg == 1:
                assert v["counts"][1] == 3
            assert v["loss_err"] <= 1e-13, (rank, agg, v)
            assert v["dz_equal"] and v["s_equal"], (rank, agg, v)
