"""GPU parity of the weight operators beyond CIS / TIS / EXACT (Table 8 and the
two-sided band of Sec. 4.3) against the fp64 oracle, through every entry point
that applies a weight: cis_weights, the fused pass (row-wise and cluster
kernels), the host-buffer path and the LM head.

Decision bands.  The band, IcePop and KPop decide in fp64 on both sides, but
with different fp64 log/exp implementations; on shared fp32 inputs a decision
may differ only where the decided quantity is within 1e-9 of its boundary.
Through the fused pass log p itself carries the GPU's fp32 error (2e-5 plus 4
ulps), so a token's decision may differ within 4e-5 of a boundary in log k; a
response's log K sums its tokens' errors, so its band is 4e-5 per token.
Tokens inside a band are left out of the weight comparison; the seeded inputs
put none there (the tests report the count and require the loss to match when
it is zero).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from _util import logits_for_oracle
from paper_2609_32444_gb300 import binding, synth
from test_gpu_parity import (DEV, TOL_LOSS, TOL_W, check_dz, check_stats, lp_tol, to_dev)

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

NEW = ["band", "icepop", "kpop", "seq_tis", "seq_mis"]
OMODE = {"band": oracle.MODE_BAND, "icepop": oracle.MODE_ICEPOP, "kpop": oracle.MODE_KPOP,
         "seq_tis": oracle.MODE_SEQ_TIS, "seq_mis": oracle.MODE_SEQ_MIS,
         "cis": oracle.MODE_CIS}
SEQ = ("seq_tis", "seq_mis")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def _kpop_metric(lw, li):
    lo, hi = 1e-8, 1.0 - 1e-8
    p = np.clip(np.exp(lw), lo, hi)
    q = np.clip(np.exp(li), lo, hi)
    with np.errstate(divide="ignore", invalid="ignore"):
        kpq = p * np.log(p / q) + (1 - p) * np.log((1 - p) / (1 - q))
        kqp = q * np.log(q / p) + (1 - q) * np.log((1 - q) / (1 - p))
    return np.maximum(kpq, kqp)


def token_band(mode, lw, li, width, lam=2.3, kappa=5e-3):
    """Tokens whose decided quantity is within `width` of a boundary."""
    lw = np.asarray(lw, np.float64)
    li = np.asarray(li, np.float64)
    logk = lw - li
    with np.errstate(invalid="ignore", divide="ignore"):
        if mode == "band":
            up = np.log1p(lam * np.maximum(-np.expm1(lw), kappa))
            low = np.log(0.5 * (1 + np.exp(lw)))
            d = np.minimum(np.abs(logk - up), np.abs(logk - low))
        elif mode == "icepop":
            d = np.minimum(np.abs(logk - math.log(0.5)), np.abs(logk - math.log(5.0)))
        elif mode == "kpop":
            d = np.abs(_kpop_metric(lw, li) - 2.0)
        elif mode == "cis":
            d = np.abs(logk - np.log1p(lam * np.maximum(-np.expm1(lw), kappa)))
        else:
            d = np.full(logk.shape, np.inf)
    return d < width


def response_band(mode, logk, mask, cu, per_token):
    """Tokens of responses whose log K is within per_token * (valid tokens) of
    a sequence boundary."""
    out = np.zeros(len(logk), bool)
    bounds = [math.log(2.0)] if mode == "seq_tis" else [math.log(0.5), math.log(2.0)]
    for i in range(len(cu) - 1):
        sl = slice(cu[i], cu[i + 1])
        v = mask[sl].astype(bool)
        LK = logk[sl][v].sum()
        if min(abs(LK - b) for b in bounds) < per_token * max(1, v.sum()):
            out[sl] = True
    return out


# ----------------------------------------------------------- cis_weights
@pytest.mark.parametrize("mode", ["band", "icepop", "kpop"])
def test_token_operators_on_shared_fp32_inputs(mode):
    """fp32 (log p, log q) pairs across confidence levels, plus pairs placed on
    the operator's boundaries: weights within 1e-5 relative, decisions equal
    except within 1e-9 of a boundary (fp64 library differences)."""
    rng = np.random.default_rng(11)
    n = 200_000
    lw = -np.exp(rng.uniform(np.log(1e-9), np.log(15.0), n))
    li = np.minimum(lw + rng.standard_normal(n) * np.where(rng.random(n) < 0.1, 3.0, 0.5),
                    -1e-12)
    if mode == "icepop":  # exactly on the bounds
        li[:1000] = lw[:1000] - math.log(0.5)
        li[1000:2000] = lw[1000:2000] - math.log(5.0)
    if mode == "band":  # exactly where e^eps = 1/2
        p = np.exp(lw[:2000])
        li[:2000] = lw[:2000] - np.log(0.5 * (1 + p))
    lw32, li32 = lw.astype(np.float32), np.minimum(li, -1e-30).astype(np.float32)
    specials_w = np.array([0.0, 0.0, -1e-30, -88.0, -np.inf, np.nan, -1.0], np.float32)
    specials_i = np.array([0.0, -1e-3, -2e-38, -1.0, -1.0, -1.0, np.nan], np.float32)
    lw32 = np.concatenate([lw32, specials_w])
    li32 = np.concatenate([li32, specials_i])
    P = binding.cis_default_params(mode)
    w, tr, _ = binding.cis_weights(torch.from_numpy(lw32).to(DEV), torch.from_numpy(li32).to(DEV),
                                   P)
    rw, rtr, _, _ = oracle.weights(lw32.astype(np.float64), li32.astype(np.float64),
                                   oracle.params(mode=OMODE[mode]))
    w, tr = w.cpu().numpy().astype(np.float64), tr.cpu().numpy()
    band = token_band(mode, lw32, li32, 1e-9)
    assert not np.any((tr != rtr) & ~band), f"{((tr != rtr) & ~band).sum()} decisions differ"
    same = (tr == rtr)
    assert np.array_equal(np.isnan(w[same]), np.isnan(rw[same]))
    fin = same & np.isfinite(rw)
    assert np.all(np.abs(w[fin] - rw[fin]) <= TOL_W * np.abs(rw[fin]) + 1e-37)
    assert 0 < rtr.sum() < len(rtr)


@pytest.mark.parametrize("mode", SEQ)
def test_sequence_operators_cis_weights(mode):
    """Responses of 1 to 300 tokens with masked tokens inside and tokens outside
    every response: each token gets its response's weight; decisions equal
    away from 1e-9 of a boundary in log K."""
    rng = np.random.default_rng(12)
    lens = rng.integers(1, 300, 400)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1]) + 50  # 50 tokens after the last response
    lw = np.log(rng.uniform(0.05, 1.0, T)).astype(np.float32)
    scale = np.repeat(rng.uniform(0.0, 0.1, len(lens)), lens)
    li = (lw.astype(np.float64) - np.concatenate([rng.standard_normal(cu[-1]) * scale,
                                                   np.zeros(50)])).astype(np.float32)
    mask = (rng.random(T) > 0.05).astype(np.uint8)
    P = binding.cis_default_params(mode)
    w, tr, _ = binding.cis_weights(torch.from_numpy(lw).to(DEV), torch.from_numpy(li).to(DEV), P,
                                   mask=torch.from_numpy(mask).to(DEV),
                                   cu_seqlens=torch.from_numpy(cu).to(DEV))
    rw, rtr, rlk, _ = oracle.weights(lw.astype(np.float64), li.astype(np.float64),
                                     oracle.params(mode=OMODE[mode]), mask=mask, cu_seqlens=cu)
    w, tr = w.cpu().numpy().astype(np.float64), tr.cpu().numpy()
    band = response_band(mode, rlk, mask, cu, 1e-12)
    assert not np.any((tr != rtr) & ~band)
    ok = ~band
    assert np.all(np.abs(w[ok] - rw[ok]) <= TOL_W * np.abs(rw[ok]) + 1e-37)
    assert np.all(w[cu[-1]:] == 0) and not tr[cu[-1]:].any()
    assert 0 < rtr.sum() < len(rtr)


# ----------------------------------------------------------- fused pass
def _check(out, ref, b, mode, lp_old=None, width=4e-5, rows_dz=None):
    mask = b.mask.cpu().numpy().astype(bool)
    lp = out["lp"].cpu().numpy().astype(np.float64)
    w = out["w"].cpu().numpy().astype(np.float64)
    tr = out["trunc"].cpu().numpy()
    ok = ~np.isnan(ref["lp"])
    assert np.all(np.abs(lp[ok] - ref["lp"][ok]) <= lp_tol(ref["lp"][ok]))
    lw = ref["lp"] if lp_old is None else lp_old.cpu().numpy().astype(np.float64)
    li = b.lp_infer.cpu().numpy()
    if mode in SEQ:
        band = response_band(mode, lw - li, b.mask.cpu().numpy(), b.cu_seqlens.cpu().numpy(),
                             width if lp_old is None else 1e-12)
    else:
        band = token_band(mode, lw, li, width if lp_old is None else 1e-9, lam=b.lam)
    good = ok & ~band
    assert not np.any((tr != ref["trunc"]) & good)
    assert np.all(np.abs(w[good] - ref["w"][good]) <= TOL_W * np.abs(ref["w"][good]) + 1e-30)
    assert np.all(w[~mask] == 0) and not tr[~mask].any()
    if not band.any():
        loss = float(out["loss"].cpu()[0])
        assert abs(loss - ref["loss"]) <= TOL_LOSS * np.abs(ref["terms"]).sum() + 1e-300
        check_stats(out["stats"], ref, li, lp_old=None if lp_old is None else
                    lp_old.cpu().numpy(), band=band, tr_gpu=tr)
        if rows_dz is None:
            check_dz(out["dlogits"], ref["dz"], ref["c"])
        else:
            check_dz(out["dlogits"][torch.from_numpy(rows_dz).to(DEV)], ref["dz"],
                     ref["c"][rows_dz])
    return int(band.sum())


def _run(b, g, mode, dz_dtype=torch.float32, lp_old=None):
    P = binding.cis_default_params(mode, lam=b.lam)
    return binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, lp_old=lp_old,
                                    mask=g["mask"], cu_seqlens=g["cu"], dlogits_dtype=dz_dtype)


def _oracle(b, mode, lp_old=None, rows=None):
    return oracle.loss_fwd_bwd(
        logits_for_oracle(b.logits), b.ids.cpu().numpy(), b.lp_infer.cpu().numpy(),
        b.adv.cpu().numpy(), oracle.params(mode=OMODE[mode], lam=b.lam),
        lp_old=None if lp_old is None else lp_old.cpu().numpy(), mask=b.mask.cpu().numpy(),
        cu_seqlens=b.cu_seqlens.cpu().numpy(), rows=rows)


@pytest.mark.parametrize("dz_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("mode", NEW)
def test_fused_pass_tiny_workload(mode, dz_dtype):
    """T=256 (4 responses of 64), V=1024, fp32 logits: every element.  The
    sequence operators run the forward pass, the response weights, then the
    pass with those weights."""
    b = synth.make_batch(1)
    g = to_dev(b)
    out = _run(b, g, mode, dz_dtype)
    ref = _oracle(b, mode)
    torch.cuda.synchronize()
    assert _check(out, ref, b, mode) == 0
    assert binding.device_status(out["workspace"]) == 0


@pytest.mark.parametrize("mode", NEW)
def test_fused_pass_with_old_logprobs(mode):
    """With l_old the weights come from it (sequence operators: formed before
    the single pass) and the PPO clip acts; every element."""
    b = synth.make_batch(1)
    g = to_dev(b)
    base = _oracle(b, "cis")
    rng = np.random.default_rng(3)
    lp_old = torch.from_numpy((base["lp"] - rng.choice([-0.3, 0.0, 0.25], size=b.T))
                              .astype(np.float32))
    out = _run(b, g, mode, lp_old=lp_old.to(DEV))
    ref = _oracle(b, mode, lp_old=lp_old)
    torch.cuda.synchronize()
    assert _check(out, ref, b, mode, lp_old=lp_old) == 0


@pytest.mark.parametrize("mode", ["band", "kpop", "seq_tis", "seq_mis"])
def test_fused_pass_cluster_path_v151936(mode):
    """48 rows of the V=151936 recipe (the 4-CTA cluster kernel), bf16 dlogits."""
    b = synth.make_batch(3, device=DEV, T=48)
    g = to_dev(b)
    out = _run(b, g, mode, torch.bfloat16)
    ref = _oracle(b, mode)
    torch.cuda.synchronize()
    assert _check(out, ref, b, mode) == 0


def test_sequence_operator_bad_id_left_out_of_the_product():
    """A token with an out-of-range id is reported and left out of its
    response's product (the other tokens' weights are unchanged)."""
    b = synth.make_batch(1)
    b.ids[5] = b.V + 3
    g = to_dev(b)
    out = _run(b, g, "seq_tis")
    ref = _oracle(b, "seq_tis")
    torch.cuda.synchronize()
    assert binding.device_status(out["workspace"]) & binding.CIS_ERR_BAD_TOKEN_ID
    w = out["w"].cpu().numpy().astype(np.float64)
    keep = np.ones(b.T, bool)
    keep[5] = False
    assert np.all(np.abs(w[keep] - ref["w"][keep]) <= TOL_W * np.abs(ref["w"][keep]) + 1e-30)
    assert np.isnan(out["lp"].cpu().numpy()[5])


# ----------------------------------------------------------- other entry points
# (the no-allocation entry point's case is in test_zz_no_alloc.py, collected last)
def test_host_path_sequence_operator():
    """The host-buffer path: Seq-TIS from l_old matches the oracle; without
    l_old it is refused (its weights would need every row before the first
    chunk)."""
    b = synth.make_batch(1)
    base = _oracle(b, "cis")
    lp_old = torch.from_numpy(base["lp"].astype(np.float32))
    P = binding.cis_default_params("seq_tis", lam=b.lam)
    dz = torch.empty((b.T, b.V), dtype=torch.float32).pin_memory()
    host = binding.cis_loss_fwd_bwd_host(b.logits, b.ids, b.lp_infer, b.adv, P, dz,
                                         lp_old=lp_old, mask=b.mask, cu_seqlens=b.cu_seqlens,
                                         chunk_tokens=48)
    torch.cuda.synchronize()
    ref = _oracle(b, "seq_tis", lp_old=lp_old)
    assert abs(float(host["loss"][0]) - ref["loss"]) <= TOL_LOSS * np.abs(ref["terms"]).sum()
    w = host["w"].numpy().astype(np.float64)
    assert np.all(np.abs(w - ref["w"]) <= TOL_W * np.abs(ref["w"]) + 1e-30)
    check_dz(dz, ref["dz"], ref["c"])
    with pytest.raises(RuntimeError):
        binding.cis_loss_fwd_bwd_host(b.logits, b.ids, b.lp_infer, b.adv, P, dz, mask=b.mask,
                                      cu_seqlens=b.cu_seqlens, chunk_tokens=48)


@pytest.mark.parametrize("mode", ["band", "icepop", "seq_tis"])
def test_lmhead_operators(mode):
    """The LM head with the band, IcePop and Seq-TIS (T=200 in responses from
    the recipe, V=1000, H=256): per-token outputs, loss, dH and dW."""
    b = synth.make_batch(5, T=200, V=1000, H=256)
    P = binding.cis_default_params(mode, lam=b.lam)
    out = binding.cis_lmhead_fused(b.hidden.to(DEV), b.weight.to(DEV), b.ids.to(DEV),
                                   b.lp_infer.to(DEV), b.adv.to(DEV), P, mask=b.mask.to(DEV),
                                   cu_seqlens=b.cu_seqlens.to(DEV))
    torch.cuda.synchronize()
    hb = b.hidden.contiguous().view(torch.int16).numpy().view(np.uint16)
    wb = b.weight.contiguous().view(torch.int16).numpy().view(np.uint16)
    m = b.mask.numpy()
    ref = oracle.lmhead_fwd_bwd(hb, wb, b.ids.numpy(), b.lp_infer.numpy(), b.adv.numpy(),
                                oracle.params(mode=OMODE[mode], lam=b.lam), mask=m,
                                cu_seqlens=b.cu_seqlens.numpy())
    lw = ref["lp"]
    li = b.lp_infer.numpy()
    if mode in SEQ:
        band = response_band(mode, lw - li, m, b.cu_seqlens.numpy(), 4e-5)
    else:
        band = token_band(mode, lw, li, 4e-5, lam=b.lam)
    assert not band.any()
    lp = out["lp"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(lp - ref["lp"]) <= lp_tol(ref["lp"]))
    w = out["w"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(w - ref["w"]) <= TOL_W * np.abs(ref["w"]) + 1e-30)
    assert np.array_equal(out["trunc"].cpu().numpy(), ref["trunc"])
    loss = float(out["loss"].cpu()[0])
    assert abs(loss - ref["loss"]) <= TOL_LOSS * np.abs(ref["terms"]).sum() + 1e-300
    for key, K in (("dhidden", b.V), ("dweight", b.T)):
        g = out[key].double().cpu().numpy()
        tol = (2.0 ** -8 + K * 2.0 ** -24) * ref[key + "_abs"] + 1e-30
        assert np.all(np.abs(g - ref[key]) <= tol)
