"""Token-sharded passes on one GPU: a batch split at response boundaries,
the shards' {N, G} counts (cis_count_valid) summed on the device in place of
the all-reduce, and each shard's fused pass run with the batch-wide counts
(cis_params_t.global_counts).  Each shard's dlogits must equal the batch's
rows bit for bit (the same arithmetic per row), and the shards' losses must
add up to the batch loss (two fp64 sums of the same terms)."""
import numpy as np
import pytest
import torch

from paper_2609_32444_gb300 import binding, shard, synth

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
