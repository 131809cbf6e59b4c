"""Token-sharded passes: a batch split at response boundaries, the shards'
{N, G} counts (cis_count_valid) summed into the batch's, and each shard's fused
pass run with the batch-wide counts (cis_params_t.global_counts).

  - Two processes on the one GPU, each a gloo rank, run
    shard.sharded_loss_fwd_bwd on their shards, so its two all-reduces (the
    counts before the pass, the loss after it) really execute.  Each rank's
    outputs are compared with the oracle's rows of the whole batch (the
    oracle given the batch's counts), and the reduced loss with the oracle's
    batch loss.  The ranks' kernels never wait on one another: the only
    exchange is gloo's, on the host, between launches.
  - In one process, the shards' counts are summed on the device in place of
    the all-reduce; each shard's dlogits must equal the batch's rows bit for
    bit (the same arithmetic per row), and the shards' losses must add up to
    the batch loss.
"""
import os
import socket
import sys
import traceback

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

from paper_2609_32444_gb300 import binding, shard, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def _batch():
    b = synth.make_batch(2, T=3000)
    mask = b.mask.clone()
    mask[::11] = 0
    cu = b.cu_seqlens.tolist()
    mask[cu[3]:cu[4]] = 0  # a response with no valid token
    return b, mask, cu


def test_count_valid_matches_numpy():
    b, mask, cu = _batch()
    got = binding.cis_count_valid(b.T, mask=mask.to(DEV),
                                  cu_seqlens=torch.tensor(cu, dtype=torch.int32, device=DEV))
    m = mask.numpy()
    n = int(m.sum())
    g = sum(1 for a, c in zip(cu, cu[1:]) if m[a:c].sum() > 0)
    assert got.cpu().tolist() == [n, g]
    assert binding.cis_count_valid(7).cpu().tolist() == [7, 0]  # no mask, no responses


@pytest.mark.parametrize("world", [2, 3])
@pytest.mark.parametrize("agg", [0, 1])
@pytest.mark.parametrize("dz", [torch.float32, torch.bfloat16])
def test_shards_reproduce_the_batch(world, agg, dz):
    b, mask, cu = _batch()
    g = dict(logits=b.logits.to(DEV), ids=b.ids.to(DEV), lp=b.lp_infer.to(DEV),
             adv=b.adv.to(DEV), mask=mask.to(DEV))
    P = binding.cis_default_params("cis", lam=b.lam, agg=agg)
    cu_dev = torch.tensor(cu, dtype=torch.int32, device=DEV)
    full = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                    cu_seqlens=cu_dev, dlogits_dtype=dz)
    parts = shard.split_at_responses(cu, world, T=b.T)
    cus = [torch.tensor(shard.shard_cu_seqlens(cu, t0, i0, i1), dtype=torch.int32, device=DEV)
           for t0, t1, i0, i1 in parts]
    counts = [binding.cis_count_valid(t1 - t0, mask=g["mask"][t0:t1], cu_seqlens=c)
              for (t0, t1, _, _), c in zip(parts, cus)]
    total = torch.stack(counts).sum(dim=0)  # what the all-reduce gives
    Pg = binding.with_global_counts(P, total)
    loss = 0.0
    for (t0, t1, _, _), c in zip(parts, cus):
        out = binding.cis_loss_fwd_bwd(g["logits"][t0:t1], g["ids"][t0:t1], g["lp"][t0:t1],
                                       g["adv"][t0:t1], Pg, mask=g["mask"][t0:t1], cu_seqlens=c,
                                       dlogits_dtype=dz)
        torch.cuda.synchronize()
        assert torch.equal(out["dlogits"], full["dlogits"][t0:t1])
        assert torch.equal(out["w"], full["w"][t0:t1])
        loss += float(out["loss"].cpu()[0])
    torch.cuda.synchronize()
    terms = (full["w"].double() * g["adv"].double()).abs().sum().item() / max(1, int(total[0]))
    assert abs(loss - float(full["loss"].cpu()[0])) <= 1e-12 * max(terms, 1e-30)
    m = mask.numpy()
    assert total.cpu().tolist() == [int(m.sum()),
                                    sum(1 for a, c in zip(cu, cu[1:]) if m[a:c].sum() > 0)]


def test_sharded_entry_point_single_rank():
    """sharded_loss_fwd_bwd on one rank (no process group) is the plain pass."""
    b, mask, cu = _batch()
    g = dict(logits=b.logits.to(DEV), ids=b.ids.to(DEV), lp=b.lp_infer.to(DEV),
             adv=b.adv.to(DEV), mask=mask.to(DEV))
    P = binding.cis_default_params("cis", lam=b.lam)
    a = shard.sharded_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                   dlogits_dtype=torch.float32)
    r = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                 dlogits_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.equal(a["dlogits"], r["dlogits"])
    assert float(a["loss"].cpu()[0]) == float(r["loss"].cpu()[0])
    assert a["global_counts"].cpu().tolist()[0] == int(mask.sum())


def _free_port():
    with socket.socket() as so:
        so.bind(("127.0.0.1", 0))
        return so.getsockname()[1]


def _rank_worker(rank, world, port, q):
    """One gloo rank: its shard through shard.sharded_loss_fwd_bwd, checked
    against the oracle's rows of the whole batch."""
    try:
        sys.path.insert(0, ROOT)
        sys.path.insert(0, os.path.join(ROOT, "tests"))
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                          WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
        import torch.distributed as dist

        import oracle
        from _util import logits_for_oracle
        from test_gpu_parity import TOL_LOSS, check_dz, check_token_outputs
        torch.cuda.set_device(0)
        dev = torch.device("cuda", 0)
        dist.init_process_group("gloo", rank=rank, world_size=world)
        try:
            b = synth.make_batch(2, T=1200, V=4096)
            mask = b.mask.clone()
            mask[::11] = 0
            cu = b.cu_seqlens.tolist()
            mask[cu[3]:cu[4]] = 0  # a response with no valid token
            m = mask.numpy()
            N = int(m.sum())
            G = sum(1 for a, c in zip(cu, cu[1:]) if m[a:c].sum() > 0)
            t0, t1, i0, i1 = shard.split_at_responses(cu, world, T=b.T)[rank]
            cu_l = shard.shard_cu_seqlens(cu, t0, i0, i1)
            g = dict(logits=b.logits[t0:t1].to(dev), ids=b.ids[t0:t1].to(dev),
                     lp=b.lp_infer[t0:t1].to(dev), adv=b.adv[t0:t1].to(dev),
                     mask=mask[t0:t1].to(dev),
                     cu=torch.tensor(cu_l, dtype=torch.int32, device=dev))
            bsub = synth.Batch(2, t1 - t0, b.V, b.logits[t0:t1], b.ids[t0:t1],
                               b.lp_infer[t0:t1], b.adv[t0:t1], mask[t0:t1],
                               torch.tensor(cu_l, dtype=torch.int32), b.lam)
            z_full = logits_for_oracle(b.logits)
            done = []
            for agg in (0, 1):
                full = oracle.loss_fwd_bwd(z_full, b.ids.numpy(), b.lp_infer.numpy(),
                                           b.adv.numpy(), oracle.params(lam=b.lam, agg=agg),
                                           mask=m, cu_seqlens=np.array(cu, np.int32),
                                           want_dz=False)
                Po = oracle.params(lam=b.lam, agg=agg, n_global=N, g_global=G)
                ref = oracle.loss_fwd_bwd(z_full[t0:t1], b.ids[t0:t1].numpy(),
                                          b.lp_infer[t0:t1].numpy(), b.adv[t0:t1].numpy(), Po,
                                          mask=m[t0:t1], cu_seqlens=np.array(cu_l, np.int32))
                # the shard's rows of the batch: the same c_t as the whole batch's
                assert np.array_equal(ref["c"], full["c"][t0:t1])
                for dz in (torch.float32, torch.bfloat16):
                    P = binding.cis_default_params("cis", lam=b.lam, agg=agg)
                    out = shard.sharded_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"],
                                                     P, mask=g["mask"], cu_seqlens=g["cu"],
                                                     dlogits_dtype=dz)
                    torch.cuda.synchronize()
                    assert out["global_counts"].cpu().tolist() == [N, G]
                    local = dict(out, loss=out["local_loss"])
                    check_token_outputs(local, ref, bsub, "cis", b.lam)
                    check_dz(out["dlogits"], ref["dz"], ref["c"])
                    loss = float(out["loss"].cpu()[0])
                    assert abs(loss - full["loss"]) <= TOL_LOSS * np.abs(full["terms"]).sum()
                    done.append((agg, str(dz)))
        finally:
            dist.destroy_process_group()
        q.put((rank, "ok", done))
    except BaseException:  # report to the parent, which asserts
        q.put((rank, traceback.format_exc(), None))


def test_two_gloo_ranks_run_the_sharded_pass_against_the_oracle():
    """Two processes (ranks over gloo) share the GPU, each running
    shard.sharded_loss_fwd_bwd on its half of a batch with masked tokens and a
    fully masked response: the all-reduced {N, G} are the batch's, each rank's
    log p, w, flags, statistics and dlogits (fp32 and bf16) match the oracle's
    rows of the batch, and the all-reduced loss matches the oracle's batch
    loss, for the token-mean (Algorithm 1) and sequence-mean (Eq. 1)
    normalisers."""
    import oracle
    oracle.build()  # once, before the ranks load it
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=600) for _ in procs)
    for p in procs:
        p.join(timeout=120)
    for rank, status, done in res:
        assert status == "ok", f"rank {rank}:\n{status}"
        assert len(done) == 4
    assert all(p.exitcode == 0 for p in procs)
