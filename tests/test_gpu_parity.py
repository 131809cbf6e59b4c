"""GPU parity: libcis (through its C ABI) against the fp64 oracle.

Tolerances (fixed by the requirements of the token pass; readings where they
need one):
  - log p of the sampled token: 2e-5 absolute, plus 4 fp32 ulps of |log p|
    (the output is fp32: the workloads' logits reach |z| ~ 650, so log p reaches
    ~ -1200, where one fp32 step is 1.2e-4; internally the weight uses log p
    carried to better than fp32 (an fp32 pair, or p = 1/(1 + t) directly in the
    fused pass's common case), so the weight tolerance below is not widened);
  - weights: 1e-5 relative;
  - truncation decisions: bit-exact when both sides get the same fp32 log-probs
    (cis_weights); end to end, bit-exact except for tokens whose fp64 log k lies
    within 4e-5 of log cap, where the fp32 log p of the GPU may legitimately
    fall on the other side (those are counted; none is expected);
  - loss: 1e-5 relative to sum_t |term_t| (the loss is a signed sum whose
    terms cancel; the bound is relative to the terms' scale);
  - fp32 dlogits: 1e-6 absolute for rows with |c_t| <= 1 and 1e-6 |c_t| above
    (dz_tj lies in [-|c_t|, |c_t|]); bf16 dlogits: at most 1 bf16 step from the
    oracle's value rounded once to bf16 (nearest, ties to even);
  - batch statistics (App. D's logged counts, Lemma B.2's excess): n_valid
    exact; n_truncated exact, or off by at most the number of tokens inside
    the decision band; max |log k| within the largest per-token error of
    log k = l_w - l_inf (the log p tolerance of l_w, plus an fp32 rounding of
    the difference); the excess within the per-token error of k (that log
    error, times k) and of w (1e-5 relative), summed over the tokens either
    side flags, plus BAND k for each token whose decision differs.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from _util import bf16_bits_from_f64, bf16_tensor_bits, bf16_ulp_distance, logits_for_oracle
from paper_2609_32444_gb300 import binding, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = torch.device("cuda")
TOL_LP, TOL_W, TOL_LOSS, TOL_DZ32, BAND = 2e-5, 1e-5, 1e-5, 1e-6, 4e-5
MODE_ID = {"cis": oracle.MODE_CIS, "tis": oracle.MODE_TIS, "exact": oracle.MODE_EXACT,
           "none": oracle.MODE_NONE}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def to_dev(b: synth.Batch):
    return {k: (None if v is None else v.to(DEV)) for k, v in
            dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv, mask=b.mask,
                 cu=b.cu_seqlens).items()}


def run_gpu(g, mode, lam, dz_dtype, lp_old=None, agg=0, use_mask=True, use_cu=False, V=None):
    P = binding.cis_default_params(mode, lam=lam, agg=agg)
    return binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, lp_old=lp_old,
                                    mask=g["mask"] if use_mask else None,
                                    cu_seqlens=g["cu"] if (use_cu or agg) else None,
                                    dlogits_dtype=dz_dtype, V=V)


def run_oracle(b, mode, lam, rows=None, lp_old=None, agg=0, use_mask=True, want_dz=True,
               logits_np=None, V=None):
    z = logits_for_oracle(b.logits) if logits_np is None else logits_np
    return oracle.loss_fwd_bwd(
        z, b.ids.cpu().numpy(), b.lp_infer.cpu().numpy(), b.adv.cpu().numpy(),
        oracle.params(mode=MODE_ID[mode], lam=lam, agg=agg), V=V,
        lp_old=None if lp_old is None else lp_old.cpu().numpy(),
        mask=b.mask.cpu().numpy() if use_mask else None,
        cu_seqlens=b.cu_seqlens.cpu().numpy() if agg else None, rows=rows, want_dz=want_dz)


def lp_tol(ref_lp):
    """2e-5 absolute plus 4 fp32 ulps of the value (2^-21 |lp| >= 4 ulp)."""
    return TOL_LP + 2.0 ** -21 * np.abs(ref_lp)


def decision_band(ref, lp_inf, mode, lam, kappa=5e-3, lp_old=None):
    """Tokens whose fp64 log k is within BAND of a truncation boundary."""
    lw = ref["lp"] if lp_old is None else lp_old.astype(np.float64)
    logk = lw - lp_inf.astype(np.float64)
    if mode == "cis":
        with np.errstate(invalid="ignore", divide="ignore"):
            dist = np.abs(logk - np.log1p(lam * np.maximum(-np.expm1(lw), kappa)))
    elif mode == "tis":
        dist = np.abs(logk - math.log(2.0))
    elif mode == "exact":
        dist = np.minimum(np.abs(logk - math.log(1e6)), np.abs(logk - math.log(1e-6)))
    else:
        dist = np.full(logk.shape, np.inf)
    return dist < BAND


def check_stats(stats_dev, ref, lp_inf, lp_old=None, band=None, tr_gpu=None):
    """The device cis_stats_t against the oracle's batch statistics.  `band`
    marks tokens whose decision may legitimately differ; `tr_gpu` is the
    GPU's per-token flag (needed when the band is not empty)."""
    st = binding.decode_stats(stats_dev)
    rs = ref["stats"]
    assert st["n_valid"] == rs["n_valid"]
    nb = 0 if band is None else int(band.sum())
    assert abs(st["n_truncated"] - rs["n_truncated"]) <= nb
    if nb == 0:
        assert st["n_truncated"] == rs["n_truncated"]
    li = np.asarray(lp_inf, np.float64)
    lw = ref["lp"] if lp_old is None else np.asarray(lp_old, np.float64)
    lk = ref["logk"]
    num = np.isfinite(lk)
    # log k error: l_w's (none when l_old is given) plus one rounding of l_w - l_inf
    lw_err = np.zeros_like(lw) if lp_old is not None else \
        TOL_LP + 2.0 ** -21 * np.abs(np.nan_to_num(lw))
    lk_err = lw_err + 2.0 ** -23 * (np.abs(np.nan_to_num(lk)) + 1e-30)
    tol_max = float(lk_err[num].max()) if num.any() else 0.0
    assert abs(st["max_abs_logk"] - rs["max_abs_logk"]) <= tol_max + 1e-30
    tr_ref = ref["trunc"].astype(bool)
    flagged = tr_ref if tr_gpu is None else (tr_ref | np.asarray(tr_gpu).astype(bool))
    flipped = np.zeros_like(tr_ref) if tr_gpu is None else \
        (tr_ref != np.asarray(tr_gpu).astype(bool))
    with np.errstate(over="ignore", invalid="ignore"):
        k = np.exp(lk)
        per = k * np.expm1(1.01 * lk_err) + TOL_W * np.abs(ref["w"]) + BAND * 1.01 * k * flipped
    want = rs["trunc_excess"]
    if not np.isfinite(want):
        assert st["trunc_excess"] == want
    else:
        tol = float(per[flagged & num].sum())
        assert abs(st["trunc_excess"] - want) <= tol + 1e-300, \
            f"excess {st['trunc_excess']} vs {want} (tol {tol})"
    return st


def check_token_outputs(out, ref, b, mode, lam, lp_old=None, use_mask=True):
    mask = b.mask.cpu().numpy().astype(bool) if use_mask else np.ones(b.T, bool)
    lp = out["lp"].cpu().numpy().astype(np.float64)
    w = out["w"].cpu().numpy().astype(np.float64)
    tr = out["trunc"].cpu().numpy()
    nan_rows = np.isnan(ref["lp"])
    assert np.array_equal(np.isnan(lp), nan_rows)
    ok = ~nan_rows
    assert np.all(np.abs(lp[ok] - ref["lp"][ok]) <= lp_tol(ref["lp"][ok]))
    wr = ref["w"][ok]
    assert np.all(np.abs(w[ok] - wr) <= TOL_W * np.abs(wr) + 1e-30)
    band = decision_band(ref, b.lp_infer.cpu().numpy(), mode, lam,
                         lp_old=None if lp_old is None else lp_old.cpu().numpy())
    mismatch = (tr != ref["trunc"]) & ~band
    assert not mismatch.any(), f"{mismatch.sum()} truncation decisions differ outside the band"
    assert not np.any(tr[~mask]) and np.all(w[~mask] == 0)
    if "stats" in out:
        check_stats(out["stats"], ref, b.lp_infer.cpu().numpy(),
                    lp_old=None if lp_old is None else lp_old.cpu().numpy(), band=band,
                    tr_gpu=tr)
    loss = float(out["loss"].cpu()[0])
    if np.isnan(ref["loss"]):
        assert np.isnan(loss)
    else:
        assert abs(loss - ref["loss"]) <= TOL_LOSS * np.abs(ref["terms"]).sum() + 1e-300
    return int(band.sum())


def check_dz(dz_gpu_rows: torch.Tensor, dz_ref: np.ndarray, c_ref: np.ndarray):
    """dz_gpu_rows [n, V] on the device or host; dz_ref [n, V] fp64; c_ref [n]."""
    if dz_gpu_rows.dtype == torch.bfloat16:
        got = bf16_tensor_bits(dz_gpu_rows)
        want = bf16_bits_from_f64(dz_ref)
        nan_g = np.isnan(dz_gpu_rows.float().cpu().numpy())
        nan_w = np.isnan(dz_ref)
        assert np.array_equal(nan_g, nan_w)
        d = bf16_ulp_distance(got, want)
        # The oracle itself is exact only to its fp64 rounding: |c| 1e-13 absolute
        # (e.g. c (p - 1) cancels to 0 in fp64 once 1 - p < 1e-16, where the GPU's
        # log-odds form still carries the true value).  Within that bound the
        # oracle cannot tell the two apart.
        gv = dz_gpu_rows.float().cpu().numpy().astype(np.float64)
        within_oracle_error = np.abs(gv - dz_ref) <= 1e-13 * np.abs(c_ref)[:, None]
        bad = (d > 1) & ~within_oracle_error & ~nan_w
        assert not bad.any(), f"bf16 dlogits off by {d[bad].max()} steps at {bad.sum()} entries"
        return int((d == 1).sum())
    got = dz_gpu_rows.float().cpu().numpy().astype(np.float64)
    nan_w = np.isnan(dz_ref)
    assert np.array_equal(np.isnan(got), nan_w)
    tol = TOL_DZ32 * np.maximum(1.0, np.abs(c_ref))[:, None]
    err = np.abs(got - dz_ref)
    assert np.all(err[~nan_w] <= np.broadcast_to(tol, err.shape)[~nan_w])
    return 0


# --------------------------------------------------------------- forward only
@pytest.mark.parametrize("cfg,T,V", [(1, None, None), (2, 512, None), (3, 40, None)])
def test_token_logprobs_match_oracle(cfg, T, V):
    b = synth.make_batch(cfg, device=DEV if cfg >= 3 else "cpu", T=T, V=V)
    g = to_dev(b)
    lp, lse = binding.cis_token_logprobs(g["logits"], g["ids"], mask=g["mask"], want_lse=True)
    ref_lp, ref_lse, rc = oracle.token_logprobs(logits_for_oracle(b.logits), b.ids.cpu().numpy(),
                                                mask=b.mask.cpu().numpy())
    assert rc == 0
    torch.cuda.synchronize()
    m = b.mask.cpu().numpy().astype(bool)
    assert np.all(np.abs(lp.cpu().numpy() - ref_lp)[m] <= lp_tol(ref_lp[m]))
    assert np.all(np.abs(lse.cpu().numpy() - ref_lse)[m] <= lp_tol(ref_lse[m]))
    assert np.all(lp.cpu().numpy()[~m] == 0)


# --------------------------------------------------------------- weights
def _weight_inputs(n=200_000, seed=3):
    """fp32 (log p, log q) pairs across confidence levels, plus pairs placed
    on (and one fp32 step either side of) every decision boundary."""
    rng = np.random.default_rng(seed)
    lw = -np.exp(rng.uniform(np.log(1e-9), np.log(15.0), n))
    li = lw + rng.standard_normal(n) * np.where(rng.random(n) < 0.1, 4.0, 0.3)
    li = np.minimum(li, -1e-12)
    lw32, li32 = lw.astype(np.float32), li.astype(np.float32)
    # boundary cases: log q = log p - log cap, then nudged by 0, +-1 ulp
    k = 20_000
    bw = lw32[:k].astype(np.float64)
    caps = [np.log1p(2.3 * np.maximum(-np.expm1(bw), 5e-3)), np.full(k, math.log(2.0)),
            np.full(k, math.log(1e6)), np.full(k, math.log(1e-6))]
    extra_w, extra_i = [], []
    for cap in caps:
        for nudge in (-1, 0, 1):
            li_b = (bw - cap).astype(np.float32)
            li_b = np.nextafter(li_b, np.float32(np.inf) if nudge > 0 else np.float32(-np.inf)) \
                if nudge else li_b
            extra_w.append(lw32[:k])
            extra_i.append(np.minimum(li_b, np.float32(-1e-30)))
    lw_all = np.concatenate([lw32] + extra_w)
    li_all = np.concatenate([li32] + extra_i)
    specials_w = np.array([0.0, -1e-30, -1e-38, -88.0, -np.inf, np.nan, -1.0], np.float32)
    specials_i = np.array([-1.0, -1e-30, -2e-38, -1.0, -1.0, -1.0, np.nan], np.float32)
    return np.concatenate([lw_all, specials_w]), np.concatenate([li_all, specials_i])


@pytest.mark.parametrize("mode", ["cis", "tis", "exact", "none"])
@pytest.mark.parametrize("lam,kappa", [(2.3, 5e-3), (0.0, 5e-3), (1.0, 0.0), (1e300, 5e-3)])
def test_weights_decisions_bit_exact_on_shared_fp32_inputs(mode, lam, kappa):
    if mode != "cis" and (lam, kappa) != (2.3, 5e-3):
        pytest.skip("lambda/kappa only matter for CIS")
    lw, li = _weight_inputs()
    P = binding.cis_default_params(mode, lam=lam, kappa=kappa)
    w, tr, eps = binding.cis_weights(torch.from_numpy(lw).to(DEV), torch.from_numpy(li).to(DEV),
                                     P, want_eps=True)
    rw, rtr, _, reps = oracle.weights(lw.astype(np.float64), li.astype(np.float64),
                                      oracle.params(mode=MODE_ID[mode], lam=lam, kappa=kappa))
    w, tr, eps = w.cpu().numpy(), tr.cpu().numpy(), eps.cpu().numpy()
    assert np.array_equal(tr, rtr), f"{(tr != rtr).sum()} decisions differ"
    fin = np.isfinite(rw)
    assert np.array_equal(np.isnan(w), np.isnan(rw))
    assert np.all(np.abs(w[fin] - rw[fin]) <= TOL_W * np.abs(rw[fin]) + 1e-37)
    ok = np.isfinite(reps) & (np.abs(reps) < 1e30)
    scale = 1 + np.abs(np.log(-np.expm1(lw.astype(np.float64)[ok]))) + \
        np.abs(np.log(-np.expm1(li.astype(np.float64)[ok])))
    assert np.all(np.abs(eps[ok] - reps[ok]) <= 2e-6 * scale + 1e-6 * np.abs(reps[ok]))


def test_weights_masked_tokens_are_zero():
    lw = torch.full((64,), -0.5, device=DEV)
    li = torch.full((64,), -2.0, device=DEV)
    mask = torch.zeros(64, dtype=torch.uint8, device=DEV)
    mask[::3] = 1
    w, tr, _ = binding.cis_weights(lw, li, binding.cis_default_params(), mask=mask)
    w, tr, m = w.cpu().numpy(), tr.cpu().numpy(), mask.cpu().numpy().astype(bool)
    assert np.all(w[~m] == 0) and not tr[~m].any() and np.all(w[m] > 0)


# --------------------------------------------------------------- fused pass
@pytest.mark.parametrize("dz_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("mode", ["cis", "tis", "exact", "none"])
def test_fwd_bwd_tiny_f32_workload(mode, dz_dtype):
    """T=256, V=1024, fp32 logits, CIS threshold 1.0: every element compared."""
    b = synth.make_batch(1)
    g = to_dev(b)
    out = run_gpu(g, mode, b.lam, dz_dtype)
    ref = run_oracle(b, mode, b.lam)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, b, mode, b.lam)
    check_dz(out["dlogits"], ref["dz"], ref["c"])
    assert binding.device_status(out["workspace"]) == 0


@pytest.mark.parametrize("dz_dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("mode", ["cis", "tis"])
def test_fwd_bwd_v32000_bf16_workload(mode, dz_dtype):
    """T=4096, V=32000 bf16 with right padding: all per-token outputs and the
    loss; dlogits on 256 rows (every padding boundary row among them)."""
    b = synth.make_batch(2)
    g = to_dev(b)
    out = run_gpu(g, mode, b.lam, dz_dtype)
    cu = b.cu_seqlens.numpy()
    rng = np.random.default_rng(0)
    rows = np.unique(np.concatenate([cu[:-1], cu[1:] - 1, np.clip(cu[-1:], 0, b.T - 1),
                                     rng.integers(0, b.T, 200)]))
    rows = rows[(rows >= 0) & (rows < b.T)]
    ref = run_oracle(b, mode, b.lam, rows=rows)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, b, mode, b.lam)
    check_dz(out["dlogits"][torch.from_numpy(rows).to(DEV)], ref["dz"], ref["c"][rows])
    masked = ~b.mask.numpy().astype(bool)
    assert torch.count_nonzero(out["dlogits"][torch.from_numpy(masked).to(DEV)]).item() == 0


@pytest.mark.parametrize("dz_dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("mode", ["cis", "tis", "exact"])
def test_fwd_bwd_v151936_rows(mode, dz_dtype):
    """The V=151936 recipe (temperatures spanning p in [1e-4, 0.9999]) on 48
    rows, every element compared; this runs the 4-CTA cluster path."""
    b = synth.make_batch(3, device=DEV, T=48)
    g = to_dev(b)
    out = run_gpu(g, mode, b.lam, dz_dtype)
    ref = run_oracle(b, mode, b.lam)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, b, mode, b.lam)
    check_dz(out["dlogits"], ref["dz"], ref["c"])


def test_fwd_bwd_long_rollout_recipe_rows():
    """The long-rollout recipe (40% padding, +6 log-odds spikes) on 640 rows."""
    b = synth.make_batch(4, device=DEV, T=640)
    g = to_dev(b)
    out = run_gpu(g, "cis", b.lam, torch.bfloat16)
    rows = np.nonzero(b.extra["spike"].cpu().numpy())[0]
    rows = np.unique(np.concatenate([rows, np.arange(0, 640, 37)]))
    ref = run_oracle(b, "cis", b.lam, rows=rows)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, b, "cis", b.lam)
    check_dz(out["dlogits"][torch.from_numpy(rows).to(DEV)], ref["dz"], ref["c"][rows])


@pytest.mark.parametrize("V,dtype", [(64, torch.bfloat16), (65536, torch.bfloat16),
                                     (151936, torch.float32), (200, torch.float32)])
def test_cluster_sizes(V, dtype):
    """Rows split over 1, 2, 4 and 8 CTAs (by row size) give the oracle's results."""
    b = synth.make_edge_rows("one_hot", V=V, T=24, dtype=dtype)
    b.logits[3::4] = (torch.randn(b.logits[3::4].shape) * 3).to(dtype)
    g = to_dev(b)
    for dz_dtype in (torch.float32, torch.bfloat16):
        out = run_gpu(g, "cis", 2.3, dz_dtype)
        ref = run_oracle(b, "cis", 2.3)
        torch.cuda.synchronize()
        check_token_outputs(out, ref, b, "cis", 2.3)
        check_dz(out["dlogits"], ref["dz"], ref["c"])


@pytest.mark.parametrize("kind", ["neg_inf", "one_hot", "flat", "ties", "huge", "nan",
                                  "masked_half"])
@pytest.mark.parametrize("V", [1024, 1001])
def test_edge_rows(kind, V):
    """Edge rows on the cluster path (V=1024) and the row-streaming path (V=1001)."""
    b = synth.make_edge_rows(kind, V=V, T=16)
    g = to_dev(b)
    for dz_dtype in (torch.float32, torch.bfloat16):
        out = run_gpu(g, "cis", 2.3, dz_dtype)
        ref = run_oracle(b, "cis", 2.3)
        torch.cuda.synchronize()
        check_token_outputs(out, ref, b, "cis", 2.3)
        check_dz(out["dlogits"], ref["dz"], ref["c"])


def test_unaligned_layouts_use_the_streaming_path_correctly():
    """Row stride not a multiple of 16 bytes, and a base pointer 2 bytes off."""
    base = synth.make_batch(3, device=DEV, T=8, V=4096)
    big = torch.zeros((8, 4099), dtype=torch.bfloat16, device=DEV)
    big[:, 1:4097] = base.logits
    view = big[:, 1:4097]  # ld = 4099, base pointer off by one element
    g = to_dev(base)
    g["logits"] = view
    out = run_gpu(g, "cis", 2.3, torch.float32)
    ref = run_oracle(base, "cis", 2.3)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, base, "cis", 2.3)
    check_dz(out["dlogits"], ref["dz"], ref["c"])


@pytest.mark.parametrize("agg", [0, 1])
def test_ppo_clip_and_sequence_mean(agg):
    """l_old given: rho = exp(l - l_old) away from 1 in both directions and
    both advantage signs (clip active and inactive), with the token-mean and the
    sequence-mean normaliser of Eq. 1."""
    b = synth.make_batch(2, T=512, V=1024)
    ref0, _, _ = oracle.token_logprobs(logits_for_oracle(b.logits), b.ids.numpy())
    rng = np.random.default_rng(4)
    shift = rng.choice([-0.6, -0.1, 0.0, 0.15, 0.5], size=b.T)
    lp_old = torch.from_numpy((ref0 - shift).astype(np.float32))
    b.adv = torch.from_numpy(rng.choice([-1.5, -0.3, 0.7, 2.0], size=b.T).astype(np.float32))
    g = to_dev(b)
    out = run_gpu(g, "cis", 2.3, torch.float32, lp_old=lp_old.to(DEV), agg=agg)
    ref = run_oracle(b, "cis", 2.3, lp_old=lp_old, agg=agg)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, b, "cis", 2.3, lp_old=lp_old)
    check_dz(out["dlogits"], ref["dz"], ref["c"])


def test_masked_rows_are_not_read():
    b = synth.make_batch(2, T=256, V=2048)
    m = b.mask.numpy().astype(bool)
    b.mask[::5] = 0
    poisoned = b.logits.clone()
    poisoned[~b.mask.numpy().astype(bool)] = float("nan")
    g = to_dev(b)
    g["logits"] = poisoned.to(DEV)
    out = run_gpu(g, "cis", 2.3, torch.bfloat16)
    ref = run_oracle(b, "cis", 2.3)
    torch.cuda.synchronize()
    assert not torch.isnan(out["dlogits"]).any()
    assert not np.isnan(float(out["loss"].cpu()[0]))
    check_token_outputs(out, ref, b, "cis", 2.3)
    check_dz(out["dlogits"], ref["dz"], ref["c"])
    assert m.any()


@pytest.mark.parametrize("T,V", [(0, 1024), (1, 1024), (5, 1), (3, 8)])
def test_degenerate_shapes(T, V):
    b = synth.make_edge_rows("flat", V=max(V, 1), T=max(T, 1), dtype=torch.float32)
    if T == 0:
        g = to_dev(b)
        empty = {k: (v[:0] if v is not None and k != "cu" else v) for k, v in g.items()}
        empty["logits"] = g["logits"][:0]
        out = binding.cis_loss_fwd_bwd(empty["logits"], empty["ids"], empty["lp"], empty["adv"],
                                       binding.cis_default_params())
        torch.cuda.synchronize()
        assert float(out["loss"].cpu()[0]) == 0.0
        assert binding.decode_stats(out["stats"])["n_valid"] == 0
        return
    if V == 1:
        b.ids.zero_()
    g = to_dev(b)
    out = run_gpu(g, "cis", 2.3, torch.float32)
    ref = run_oracle(b, "cis", 2.3)
    torch.cuda.synchronize()
    check_token_outputs(out, ref, b, "cis", 2.3)
    check_dz(out["dlogits"], ref["dz"], ref["c"])


def test_out_of_range_ids_set_the_status_bit_only_for_their_rows():
    b = synth.make_batch(1, T=64)
    b.ids[5] = b.V
    b.ids[9] = -3
    g = to_dev(b)
    out = run_gpu(g, "cis", b.lam, torch.float32)
    torch.cuda.synchronize()
    assert binding.device_status(out["workspace"]) & binding.CIS_ERR_BAD_TOKEN_ID
    st = binding.decode_stats(out["stats"])
    assert st["status"] & binding.CIS_ERR_BAD_TOKEN_ID
    lp = out["lp"].cpu().numpy()
    assert np.isnan(lp[5]) and np.isnan(lp[9]) and np.isfinite(np.delete(lp, [5, 9])).all()
    dz = out["dlogits"].cpu()
    assert torch.count_nonzero(dz[5]) == 0 and torch.count_nonzero(dz[9]) == 0
    good = np.setdiff1d(np.arange(64), [5, 9])
    b.ids[5] = 0
    b.ids[9] = 0
    ref = run_oracle(b, "cis", b.lam, rows=good)
    check_dz(out["dlogits"][torch.from_numpy(good).to(DEV)], ref["dz"], ref["c"][good])


def test_deterministic_and_stream_ordered():
    b = synth.make_batch(3, device=DEV, T=64)
    g = to_dev(b)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        a1 = run_gpu(g, "cis", 2.3, torch.bfloat16)
        a2 = run_gpu(g, "cis", 2.3, torch.bfloat16)
    s.synchronize()
    assert torch.equal(a1["dlogits"].view(torch.int16), a2["dlogits"].view(torch.int16))
    assert torch.equal(a1["loss"], a2["loss"]) and torch.equal(a1["lp"], a2["lp"])


# --------------------------------------------------------------- full sizes
def _full_size_check(cfg, mode, dz_dtype, n_sample_rows=48):
    b = synth.make_batch(cfg, device=DEV)
    g = to_dev(b)
    out = run_gpu(g, mode, b.lam, dz_dtype)
    torch.cuda.synchronize()
    mask = b.mask.cpu().numpy().astype(bool)
    nvalid = int(mask.sum())
    assert mask[:nvalid].all()  # responses are packed from row 0; padding follows
    host = logits_for_oracle(b.logits[:nvalid])
    bsub = synth.Batch(cfg, nvalid, b.V, None, b.ids[:nvalid], b.lp_infer[:nvalid],
                       b.adv[:nvalid], b.mask[:nvalid], b.cu_seqlens, b.lam)
    pst = b.extra["pstar"][:nvalid].cpu().numpy()
    rng = np.random.default_rng(1)
    rows = np.unique(np.concatenate([[0, nvalid - 1, int(np.argmin(pst)), int(np.argmax(pst))],
                                     rng.integers(0, nvalid, n_sample_rows)]))
    ref = run_oracle(bsub, mode, b.lam, rows=rows, logits_np=host)
    # per-token outputs of the valid rows; the loss is a sum over valid rows only
    sub = {k: (v[:nvalid] if k in ("lp", "w", "trunc") else v) for k, v in out.items()}
    n_band = check_token_outputs(sub, ref, bsub, mode, b.lam)
    check_dz(out["dlogits"][torch.from_numpy(rows).to(DEV)], ref["dz"], ref["c"][rows])
    if nvalid < b.T:
        assert torch.count_nonzero(out["dlogits"][nvalid:]).item() == 0
    # every valid row: finite, and sum_j dz_tj = c (sum_j softmax_j - 1) = 0 up
    # to the bf16 rounding of each element (2^-9 relative, so 2^-8 of the
    # row's L1 norm bounds the sum)
    for r0 in range(0, nvalid, 2048):
        dz = out["dlogits"][r0:min(nvalid, r0 + 2048)].float()
        assert torch.isfinite(dz).all()
        assert torch.all(dz.sum(dim=1).abs() <= 2.0 ** -8 * dz.abs().sum(dim=1) + 1e-30)
    st = binding.decode_stats(out["stats"])
    assert st["n_valid"] == nvalid and st["status"] == 0
    return n_band


@pytest.mark.parametrize("mode", ["cis", "tis", "exact"])
def test_full_size_t16384_v151936(mode):
    """The benchmarked workload itself: all per-token outputs and the loss
    against the oracle over every row, dlogits on sampled rows."""
    assert _full_size_check(3, mode, torch.bfloat16) == 0


def test_full_size_t65536_v151936_masked():
    _full_size_check(4, "cis", torch.bfloat16)


@pytest.mark.parametrize("mode", ["cis", "tis", "exact", "none"])
def test_direct_weight_boundaries_v151936(mode):
    """The fused pass at V=151936 (4-CTA clusters) on rows built to sit at the
    edges of its logarithm-free common case: inference log-probs that put
    log k within 1e-7 .. 1e-3 of the operator's cap (either side, so that the
    fp32 comparison is certain for some and hands over to the fp64 fallback
    for others), z_y - m' near the +-70 range guard, and l_inf near -70.
    Decisions outside the 4e-5 band, weights, loss and every dlogits entry are
    checked against the oracle."""
    T, lam = 64, 2.3
    b = synth.make_batch(3, device=DEV, T=T)
    z = b.logits.float()
    ids = b.ids.long()
    # rows 48..55: z_y - m' just inside / outside +-70 (m' = max over j != y)
    zz = z.clone()
    zz[torch.arange(T, device=DEV), ids] = -float("inf")
    mprime = zz.max(dim=1).values
    for i, off in enumerate([69.0, -69.0, 72.0, -72.0, 69.75, -69.75, 70.5, -70.5]):
        t = 48 + i
        z[t, ids[t]] = mprime[t] + off
    b.logits = z.to(torch.bfloat16)
    z_np = logits_for_oracle(b.logits)
    ref_lp, _, _ = oracle.token_logprobs(z_np, b.ids.cpu().numpy())
    deltas = np.array([0.0, 1e-7, -1e-7, 1e-6, -1e-6, 3e-6, -3e-6, 1e-5, -1e-5, 1e-4, -1e-4,
                       1e-3, -1e-3, 5e-3, -5e-3, 2e-2])
    lp_inf = ref_lp.copy()
    for t in range(48):
        d = deltas[t % len(deltas)]
        if mode == "cis":
            logcap = np.log1p(lam * max(-np.expm1(ref_lp[t]), 5e-3))
        elif mode == "tis":
            logcap = math.log(2.0)
        elif mode == "exact":
            logcap = math.log(1e6) if t % 2 else math.log(1e-6)
        else:
            logcap = 0.0
        lp_inf[t] = ref_lp[t] - logcap - d  # log k = log cap + d
    lp_inf[56:60] = [-69.0, -71.0, -69.9, -70.1]  # around the l_inf guard
    b.lp_infer = torch.from_numpy(lp_inf.astype(np.float32))
    b.adv = torch.from_numpy(np.where(np.arange(T) % 3 == 0, -1.0, 0.75).astype(np.float32))
    g = to_dev(b)
    for dz_dtype in (torch.float32, torch.bfloat16):
        out = run_gpu(g, mode, lam, dz_dtype)
        ref = run_oracle(b, mode, lam)
        torch.cuda.synchronize()
        check_token_outputs(out, ref, b, mode, lam)
        check_dz(out["dlogits"], ref["dz"], ref["c"])
