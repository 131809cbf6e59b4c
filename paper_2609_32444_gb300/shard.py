"""Token-sharded data parallelism for the CIS token pass (one process per GPU).

The rows of a batch are independent, so a batch splits across ranks at
response boundaries and every rank runs the fused pass on its own rows.  The
only batch-wide quantity is the loss normaliser: Algorithm 1 divides by the
number of valid tokens n of the batch, Eq. 1 by the number of responses G
(and each response by its own length, which stays inside one shard).  So each
rank counts its {N, G} on the device, the ranks all-reduce the pair before
the pass, and after it they all-reduce the fp64 loss: each rank's dlogits are
exactly the batch's rows, and the losses add up to the batch loss.
"""
from __future__ import annotations

from typing import Sequence

import torch
import torch.distributed as dist

from . import binding


def split_at_responses(cu_seqlens: Sequence[int], world: int, T: int | None = None):
    """Split responses [cu[i], cu[i+1]) into `world` contiguous shards of about
    equal token counts, cutting only at response boundaries.  Returns, per
    rank, (t0, t1, i0, i1): rows [t0, t1) and responses [i0, i1).  Rows after
    the last response (padding) go to the last shard when T is given."""
    cu = [int(c) for c in cu_seqlens]
    if world < 1 or len(cu) < 1 or any(b < a for a, b in zip(cu, cu[1:])):
        raise ValueError("need world >= 1 and a non-decreasing cu_seqlens")
    B = len(cu) - 1
    total = cu[-1] - cu[0]
    cuts = [0]
    for r in range(1, world):
        target = cu[0] + total * r / world
        # the response boundary closest to the target, not before the last cut
        i = min(range(cuts[-1], B + 1), key=lambda k: (abs(cu[k] - target), k))
        cuts.append(i)
    cuts.append(B)
    shards = []
    for r in range(world):
        i0, i1 = cuts[r], cuts[r + 1]
        t0 = cu[i0] if r > 0 else 0
        t1 = cu[i1] if r < world - 1 else (cu[-1] if T is None else max(T, cu[-1]))
        shards.append((t0, t1, i0, i1))
    return shards


def shard_cu_seqlens(cu_seqlens: Sequence[int], t0: int, i0: int, i1: int) -> list[int]:
    """The shard's own cu_seqlens (rows counted from t0)."""
    return [int(c) - t0 for c in cu_seqlens[i0:i1 + 1]]


def sharded_loss_fwd_bwd(logits: torch.Tensor, ids: torch.Tensor, lp_infer: torch.Tensor,
                         adv: torch.Tensor, params: binding.cis_params_t, mask=None,
                         cu_seqlens=None, group=None, **kw):
    """This rank's fused pass over its shard of a batch.  Before the pass the
    ranks all-reduce their {N, G} (cis_count_valid) into the normaliser the
    pass uses; after it they all-reduce the fp64 loss, so out["loss"] is the
    batch loss on every rank and out["dlogits"] are this shard's rows of the
    batch's gradient.  out["local_loss"] keeps this shard's share, and
    out["stats"] stays per shard.  Keyword arguments go to cis_loss_fwd_bwd."""
    T = logits.shape[0]
    counts = binding.cis_count_valid(T, mask=mask, cu_seqlens=cu_seqlens)
    if dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(counts, group=group)
    out = binding.cis_loss_fwd_bwd(logits, ids, lp_infer, adv,
                                   binding.with_global_counts(params, counts), mask=mask,
                                   cu_seqlens=cu_seqlens, **kw)
    out["global_counts"] = counts  # read by the pass's first kernel: kept alive with the result
    out["local_loss"] = out["loss"].clone()
    if dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(out["loss"], group=group)
    return out
