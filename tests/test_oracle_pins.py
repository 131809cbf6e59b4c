"""Pins of the fp64 oracle against what the paper and mathematics fix.

None of these compares the oracle with itself: each check is a closed form, a
special case that reduces to a textbook quantity, an identity the paper
proves, a number the paper prints (tests/golden/paper_values.json), brute
force at 50 digits, or central finite differences of the loss.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle

mpmath = pytest.importorskip("mpmath")

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


def _rng(seed):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- log-softmax
@pytest.mark.parametrize("V", [1, 2, 5, 8])
def test_logprob_tiny_v_matches_50_digit_brute_force(V):
    """log p_y = log(e^{z_y} / sum_j e^{z_j}) (Sec. 2.1), evaluated at 50 digits."""
    rng = _rng(V)
    T = 16
    z = (rng.standard_normal((T, V)) * 6).astype(np.float32)
    ids = rng.integers(0, V, T).astype(np.int32)
    lp, lse, rc = oracle.token_logprobs(z, ids)
    assert rc == 0
    mpmath.mp.dps = 50
    for t in range(T):
        num = mpmath.e ** mpmath.mpf(float(z[t, ids[t]]))
        den = mpmath.fsum(mpmath.e ** mpmath.mpf(float(v)) for v in z[t])
        ref = float(mpmath.log(num / den))
        assert abs(lp[t] - ref) <= 1e-13 * max(1.0, abs(ref))
        assert abs(lse[t] - float(mpmath.log(den))) <= 1e-13 * max(1.0, abs(float(mpmath.log(den))))


def test_logprob_shift_invariance():
    """softmax(z + c) = softmax(z): log p is unchanged by a constant shift."""
    rng = _rng(1)
    z = (rng.integers(-256, 256, (8, 300)) / 64.0).astype(np.float32)
    ids = rng.integers(0, 300, 8).astype(np.int32)
    lp0, _, _ = oracle.token_logprobs(z, ids)
    lp1, _, _ = oracle.token_logprobs(z + np.float32(3.0), ids)  # exact in fp32
    np.testing.assert_allclose(lp0, lp1, rtol=0, atol=1e-12)


def test_logsumexp_normalises():
    """sum_j exp(z_j - lse) = 1 for every row (the softmax is a distribution)."""
    rng = _rng(2)
    z = (rng.standard_normal((32, 1024)) * 4).astype(np.float32)
    ids = np.zeros(32, np.int32)
    _, lse, _ = oracle.token_logprobs(z, ids)
    tot = np.exp(z.astype(np.float64) - lse[:, None]).sum(axis=1)
    np.testing.assert_allclose(tot, 1.0, rtol=0, atol=1e-12)


def test_bf16_decoding_matches_library_conversion():
    """bf16 rows must give the same log p as the same values given as fp32."""
    torch = pytest.importorskip("torch")
    rng = _rng(3)
    zf = torch.from_numpy((rng.standard_normal((16, 77)) * 5).astype(np.float32))
    zb = zf.to(torch.bfloat16)
    bits = zb.view(torch.int16).numpy().view(np.uint16)
    ids = rng.integers(0, 77, 16).astype(np.int32)
    lp_b, _, _ = oracle.token_logprobs(bits, ids)
    lp_f, _, _ = oracle.token_logprobs(zb.float().numpy(), ids)
    np.testing.assert_array_equal(lp_b, lp_f)


def test_minus_inf_logits_and_masked_rows():
    """-inf logits contribute e^-inf = 0; masked rows are skipped (lp = 0)."""
    z = np.array([[0.0, -np.inf, math.log(3.0)], [1.0, 2.0, 3.0]], np.float32)
    ids = np.array([0, 2], np.int32)
    lp, _, rc = oracle.token_logprobs(z, ids, mask=np.array([1, 0], np.uint8))
    assert rc == 0
    ref = -math.log(1.0 + math.exp(float(z[0, 2])))  # e^0 / (e^0 + e^-inf + e^{z_2})
    assert abs(lp[0] - ref) < 1e-15
    assert lp[1] == 0.0


def test_bad_token_id_is_reported():
    z = np.zeros((2, 4), np.float32)
    lp, _, rc = oracle.token_logprobs(z, np.array([0, 4], np.int32))
    assert rc == -1 and math.isnan(lp[1]) and lp[0] == pytest.approx(-math.log(4))


# ---------------------------------------------------------------- weights
def _inference_pair(rng, V, n, scale=2.0, dscale=0.5):
    """Training logits z, inference logits z + delta, and the sampled ids."""
    z = rng.standard_normal((n, V)) * scale
    delta = rng.standard_normal((n, V)) * dscale
    ids = rng.integers(0, V, n)
    return z, delta, ids


def _log_softmax(x):
    m = x.max(axis=1, keepdims=True)
    return x - m - np.log(np.exp(x - m).sum(axis=1, keepdims=True))


def test_lemma_3_1_ratio_displacement_identity():
    """Lemma 3.1 / B.1: with eps := -delta_y + log sum_{j!=y} w_j e^{delta_j},
    w_j = e^{z_j} / sum_{j'!=y} e^{z_j'}, one has k = p + (1-p) e^eps and
    eps = logit p - logit q.  eps is computed here from the full logit
    vectors by its definition; the oracle only sees log p and log q."""
    rng = _rng(10)
    n, V = 200, 50
    z, delta, ids = _inference_pair(rng, V, n)
    lp = _log_softmax(z)[np.arange(n), ids]
    lq = _log_softmax(z + delta)[np.arange(n), ids]
    _, _, logk, eps = oracle.weights(lp, lq, oracle.params(mode=oracle.MODE_EXACT, exact_lo=0,
                                                           exact_hi=np.inf))
    eps_def = np.empty(n)
    for t in range(n):
        y = ids[t]
        others = np.arange(V) != y
        wj = np.exp(z[t, others]) / np.exp(z[t, others]).sum()
        eps_def[t] = -delta[t, y] + math.log(float((wj * np.exp(delta[t, others])).sum()))
    np.testing.assert_allclose(eps, eps_def, rtol=1e-9, atol=1e-9)
    p = np.exp(lp)
    np.testing.assert_allclose(np.exp(logk), p + (1 - p) * np.exp(eps_def), rtol=1e-9)


def test_ratio_is_one_without_perturbation_and_gauge_invariant():
    """delta = 0, or delta = const (the gauge freedom of App. A.1), gives
    q = p, k = 1, w = 1 in every mode and no truncation."""
    rng = _rng(11)
    n, V = 64, 40
    z, _, ids = _inference_pair(rng, V, n)
    lp = _log_softmax(z)[np.arange(n), ids]
    lq = _log_softmax(z + 7.25)[np.arange(n), ids]
    for mode in (oracle.MODE_CIS, oracle.MODE_TIS, oracle.MODE_EXACT, oracle.MODE_NONE):
        w, tr, logk, _ = oracle.weights(lp, lq, oracle.params(mode=mode))
        np.testing.assert_allclose(logk, 0.0, atol=1e-13)
        np.testing.assert_allclose(w, 1.0, rtol=1e-12)
        assert not tr.any()


def _random_lw_linf(rng, n):
    lw = -np.exp(rng.uniform(np.log(1e-7), np.log(12.0), n))  # log p over many decades
    linf = lw + rng.standard_normal(n) * 1.5
    linf = np.minimum(linf, -1e-9)
    return lw, linf


def test_lambda_zero_is_tis_with_cap_one():
    """lambda = 0 gives f = min(k, 1), i.e. TIS with C = 1 (Sec. 4.3/4.4)."""
    assert GOLDEN["lambda_zero_is_tis_c1"]["value"]
    rng = _rng(12)
    lw, linf = _random_lw_linf(rng, 2000)
    w, tr, _, _ = oracle.weights(lw, linf, oracle.params(lam=0.0))
    k = np.exp(lw - linf)
    np.testing.assert_allclose(w, np.minimum(k, 1.0), rtol=1e-14)
    np.testing.assert_array_equal(tr.astype(bool), lw - linf > 0)


def test_lambda_to_infinity_is_exact_ratio():
    """lambda -> inf recovers the exact ratio (Sec. 3.3, after Theorem 3.3)."""
    assert GOLDEN["lambda_inf_is_exact"]["value"]
    rng = _rng(13)
    lw, linf = _random_lw_linf(rng, 2000)
    w, tr, _, _ = oracle.weights(lw, linf, oracle.params(lam=1e300))
    np.testing.assert_allclose(w, np.exp(lw - linf), rtol=1e-14)
    assert not tr.any()


def _cap(lw, lam=2.3, kappa=5e-3):
    """The CIS cap as the weight of a token with an enormous ratio."""
    lw = np.asarray(lw, np.float64)
    w, tr, _, _ = oracle.weights(lw, lw - 800.0, oracle.params(lam=lam, kappa=kappa))
    assert tr.all()
    return w


def test_cap_monotone_in_confidence_and_floor_value():
    """cap(p) = 1 + lambda max(1-p, kappa) is non-increasing in p and equals
    1 + lambda*kappa below the floor; the paper prints that value as ~1.01."""
    p = np.linspace(1e-6, 1 - 1e-9, 20001)
    caps = _cap(np.log(p))
    assert np.all(np.diff(caps) <= 1e-15)
    lam = GOLDEN["lambda_default"]["value"]
    kap = GOLDEN["kappa_default"]["value"]
    below = caps[(1 - p) < kap]
    np.testing.assert_allclose(below, 1 + lam * kap, rtol=1e-15)
    g = GOLDEN["cap_below_floor"]
    assert round(float(below[0]), g["decimals"]) == g["value"]
    # above the floor the cap follows 1 + lambda (1 - p) (Eq. 4)
    above = (1 - p) > kap
    np.testing.assert_allclose(caps[above], 1 + lam * (1 - p[above]), rtol=1e-12)


def test_cis_cap_looser_than_tis2_below_printed_confidence():
    """The CIS cap exceeds C = 2 exactly when p < 1 - 1/lambda; the paper
    prints the crossing as p = 0.565 (Sec. 4.3)."""
    g = GOLDEN["cis_looser_than_tis2_below_p"]
    p = np.linspace(0.4, 0.7, 300001)
    caps = _cap(np.log(p))
    crossing = p[np.argmax(caps <= 2.0)]
    assert round(float(crossing), g["decimals"]) == g["value"]
    assert abs(crossing - (1 - 1 / 2.3)) < 2e-6


def test_corollary_b6_floor_ordering():
    """Corollary B.6: f_lambda <= f_{lambda,kappa} <= k and f_{lambda,kappa} <= 1 + lambda."""
    rng = _rng(14)
    lw, linf = _random_lw_linf(rng, 5000)
    k = np.exp(lw - linf)
    for lam in (0.0, 0.5, 2.3, 10.0):
        for kap in (1e-3, 5e-3, 0.1, 1.0):
            f0, _, _, _ = oracle.weights(lw, linf, oracle.params(lam=lam, kappa=0.0))
            fk, _, _, _ = oracle.weights(lw, linf, oracle.params(lam=lam, kappa=kap))
            assert np.all(f0 <= fk * (1 + 1e-15))
            assert np.all(fk <= k * (1 + 1e-15))
            assert np.all(fk <= (1 + lam) * (1 + 1e-15))


def test_lemma_b2_truncated_excess_and_one_sidedness():
    """Lemma B.2: k - f_lambda = (1-p)(e^eps - 1 - lambda)_+, and eps <= 0
    implies p < k <= 1 (eps = logit p - logit q)."""
    rng = _rng(15)
    lw, linf = _random_lw_linf(rng, 5000)
    p = np.exp(lw)
    # logit p - logit q written out from the two probabilities
    eps = (lw - np.log(-np.expm1(lw))) - (linf - np.log(-np.expm1(linf)))
    k = np.exp(lw - linf)
    for lam in (0.0, 1.0, 2.3):
        f, _, _, _ = oracle.weights(lw, linf, oracle.params(lam=lam, kappa=0.0))
        excess = (1 - p) * np.maximum(np.exp(eps) - 1 - lam, 0.0)
        assert np.all(np.abs((k - f) - excess) <= 1e-8 * np.abs(excess) + 1e-12 * np.maximum(k, 1))
    neg = eps <= 0
    assert np.all(k[neg] <= 1 + 1e-15) and np.all(k[neg] > p[neg])


def test_eq5_fixed_cap_in_displacement_coordinate():
    """Eq. 5 / Lemma B.2: k <= C  <=>  e^eps <= 1 + (C-1)/(1-p)."""
    rng = _rng(16)
    lw, linf = _random_lw_linf(rng, 5000)
    p = np.exp(lw)
    eps = (lw - np.log(-np.expm1(lw))) - (linf - np.log(-np.expm1(linf)))
    for C in (1.0, 1.13, 2.0, 5.0):
        _, tr, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_TIS, tis_cap=C))
        rhs = np.exp(eps) <= 1 + (C - 1) / (1 - p)
        lk = lw - linf
        clear = np.abs(lk - math.log(C)) > 1e-9  # stay off exact ties
        np.testing.assert_array_equal((tr == 0)[clear], rhs[clear])


def test_exact_ratio_clamp_and_tis_defaults():
    """Table 8: exact ratio clamped to [1e-6, 1e6]; TIS cap C = 2."""
    lo, hi = GOLDEN["exact_clamp"]["value"]
    lw = np.array([-1.0, -1.0, -1.0, -0.1])
    linf = np.array([-30.0, -1.0 + 1e-3, 40.0, -0.1 - math.log(3.0)])
    w, tr, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_EXACT))
    assert w[0] == hi and tr[0] == 1
    assert w[1] == pytest.approx(math.exp(-1e-3)) and tr[1] == 0
    assert w[2] == lo and tr[2] == 1
    w, tr, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_TIS))
    assert w[3] == GOLDEN["tis_cap_default"]["value"] and tr[3] == 1


def test_calibration_identity_by_brute_force():
    """E_{y~q}[k_y] = sum_j q_j p_j / q_j = 1 per position (App. C.4), with
    p_j from the oracle's log-softmax over every possible sampled token."""
    rng = _rng(17)
    V = 64
    for _ in range(5):
        z = (rng.standard_normal((1, V)) * 3).astype(np.float32)
        delta = rng.standard_normal(V) * 0.7
        zz = np.repeat(z, V, axis=0)
        lp, _, _ = oracle.token_logprobs(zz, np.arange(V, dtype=np.int32))
        lq = _log_softmax((z.astype(np.float64) + delta))[0]
        _, _, logk, _ = oracle.weights(lp, lq, oracle.params(mode=oracle.MODE_NONE))
        assert abs(float((np.exp(lq) * np.exp(logk)).sum()) - 1.0) < 1e-13


# ---------------------------------------------------------------- normaliser
def test_loss_scales_token_and_sequence_mean():
    """Algorithm 1 averages over the n tokens; Eq. 1 averages each response
    over its |y_i| tokens and then over the G responses."""
    mask = np.array([1, 1, 1, 1, 1, 0, 1], np.uint8)
    s = oracle.loss_scales(7, mask)
    np.testing.assert_allclose(s, [1 / 6] * 5 + [0] + [1 / 6])
    cu = np.array([0, 1, 6], np.int32)  # response 0: token 0; response 1: tokens 1..5
    s = oracle.loss_scales(7, mask, cu, oracle.AGG_SEQ_MEAN)
    np.testing.assert_allclose(s, [1 / 2, 1 / 8, 1 / 8, 1 / 8, 1 / 8, 0, 0])


# ---------------------------------------------------------------- loss / gradient
def test_loss_closed_forms():
    """No correction, on-policy: loss = -(1/n) sum_t A_t.  A ratio of exactly 2
    with A = 1 is clipped at 1 + c_high = 1.28 (Eq. 1)."""
    rng = _rng(20)
    T, V = 12, 9
    z = (rng.integers(-64, 64, (T, V)) / 16).astype(np.float32)
    ids = rng.integers(0, V, T).astype(np.int32)
    adv = rng.standard_normal(T)
    mask = np.ones(T, np.uint8)
    mask[3] = 0
    out = oracle.loss_fwd_bwd(z, ids, np.zeros(T), adv, oracle.params(mode=oracle.MODE_NONE),
                              mask=mask, want_dz=False)
    assert out["loss"] == pytest.approx(-adv[mask == 1].sum() / 11, rel=1e-14)
    lp, _, _ = oracle.token_logprobs(z, ids)
    out = oracle.loss_fwd_bwd(z, ids, lp, np.ones(T), oracle.params(mode=oracle.MODE_NONE),
                              lp_old=lp - math.log(2.0), want_dz=True)
    assert out["loss"] == pytest.approx(-1.28, rel=1e-13)
    assert np.abs(out["dz"]).max() == 0.0  # the clip is active on every token
    out = oracle.loss_fwd_bwd(z, ids, lp, -np.ones(T), oracle.params(mode=oracle.MODE_NONE),
                              lp_old=lp - math.log(2.0), want_dz=False)
    assert out["loss"] == pytest.approx(2.0, rel=1e-13)  # A < 0: min picks rho*A = -2



# ---------------------------------------------------------------- batch statistics
def test_stats_lemma_b2_sum_and_displacement_count():
    """The batch statistics of the pass (App. D logs how many tokens the
    correction acts on and the largest |log k|; Lemma B.2 gives the ratio
    mass a capped token loses).  With kappa = 0, Lemma B.2 gives
    k - f = (1 - p)(e^eps - 1 - lambda)_+ per token, so the summed truncated
    excess is that sum over the valid tokens, and a token is truncated exactly
    when e^eps > 1 + lambda (Eq. 4's threshold).  p comes from a library
    log-softmax of the logits, eps = logit p - logit q from the two
    probabilities: neither the cap nor the truncation flag enters."""
    from scipy.special import log_softmax
    rng = _rng(70)
    T, V, lam = 400, 40, 2.3
    z = (rng.standard_normal((T, V)) * 2.5).astype(np.float32)
    ids = rng.integers(0, V, T).astype(np.int32)
    lp = log_softmax(z.astype(np.float64), axis=1)[np.arange(T), ids]
    lq = np.minimum(lp + rng.standard_normal(T) * 1.2, -1e-6)
    mask = (rng.random(T) > 0.15).astype(np.uint8)
    out = oracle.loss_fwd_bwd(z, ids, lq, rng.standard_normal(T),
                              oracle.params(lam=lam, kappa=0.0), mask=mask, want_dz=False)
    st = out["stats"]
    v = mask == 1
    p, q = np.exp(lp), np.exp(lq)
    eps = (lp - np.log1p(-p)) - (lq - np.log1p(-q))
    excess = ((1 - p) * np.maximum(np.exp(eps) - 1 - lam, 0.0))[v].sum()
    assert st["n_valid"] == int(v.sum())
    assert st["n_truncated"] == int((np.exp(eps) > 1 + lam)[v].sum())
    assert 20 < st["n_truncated"] < v.sum() - 20
    assert st["trunc_excess"] == pytest.approx(excess, rel=1e-9)
    assert st["max_abs_logk"] == pytest.approx(np.abs(lp - lq)[v].max(), rel=1e-12)
    assert np.abs(np.abs(lp - lq)[~v]).max() > 0  # masked tokens would change nothing otherwise


def _two_logit_batch(k_targets, x=0.0):
    """Rows of two logits [0, x] with the sampled id 0 (p = 1/(1 + e^x)) and
    an inference log-prob that puts the ratio k at each target."""
    T = len(k_targets)
    z = np.tile(np.array([0.0, x], np.float32), (T, 1))
    lp = -math.log1p(math.exp(x))
    lq = lp - np.log(np.asarray(k_targets, np.float64))
    return z, np.zeros(T, np.int32), lq, lp


@pytest.mark.parametrize("with_old", [False, True])
@pytest.mark.parametrize("case", ["tis", "exact", "icepop", "band", "none"])
def test_stats_hand_built_batches(case, with_old):
    """Batches with known counts: which tokens an operator changes (Table 8,
    Sec. 4.3), the excess k - w they lose (negative when the band lifts a
    token or the exact ratio is clamped from below), masked tokens and a token
    with an out-of-range id left out of everything but n_valid (with l_old
    given, that token's log k is a finite number and must still be left
    out)."""
    if case == "tis":       # C = 2
        ks, P = [3.0, 1.5, 5.0, 100.0, 0.25], oracle.params(mode=oracle.MODE_TIS)
        want = dict(n_truncated=2, trunc_excess=(3 - 2) + (5 - 2), max_abs_logk=math.log(5.0))
    elif case == "exact":   # clamp to [1e-6, 1e6]
        ks, P = [1e7, 1e-7, 2.0, 100.0, 0.5], oracle.params(mode=oracle.MODE_EXACT)
        want = dict(n_truncated=2, trunc_excess=(1e7 - 1e6) + (1e-7 - 1e-6),
                    max_abs_logk=math.log(1e7))
    elif case == "icepop":  # kept on [0.5, 5], else 0
        ks, P = [0.25, 6.0, 1.0, 100.0, 5.0], oracle.params(mode=oracle.MODE_ICEPOP)
        want = dict(n_truncated=2, trunc_excess=0.25 + 6.0, max_abs_logk=math.log(6.0))
    elif case == "band":    # p = 1/2: cap 1 + 2.3/2 = 2.15, floor (1 + 1/2)/2 = 0.75
        ks, P = [0.5, 3.0, 1.0, 100.0, 2.0], oracle.params(mode=oracle.MODE_BAND, lam=2.3)
        want = dict(n_truncated=2, trunc_excess=(0.5 - 0.75) + (3.0 - 2.15),
                    max_abs_logk=math.log(3.0))
    else:
        ks, P = [3.0, 0.1, 1.0, 100.0, 2.0], oracle.params(mode=oracle.MODE_NONE)
        want = dict(n_truncated=0, trunc_excess=0.0, max_abs_logk=math.log(10.0))
    ks = ks + [1e6]  # the last token's id is out of range
    z, ids, lq, lp = _two_logit_batch(ks)
    ids[-1] = 7
    mask = np.array([1, 1, 1, 0, 1, 1], np.uint8)  # k = 100 is masked
    lp_old = np.full(len(ks), lp) if with_old else None
    out = oracle.loss_fwd_bwd(z, ids, lq, np.ones(len(ks)), P, mask=mask, lp_old=lp_old,
                              want_dz=False)
    assert out["rc"] == -1  # the out-of-range id is reported
    st = out["stats"]
    assert st["n_valid"] == 5
    assert st["n_truncated"] == want["n_truncated"]
    assert st["trunc_excess"] == pytest.approx(want["trunc_excess"], rel=1e-12, abs=1e-15)
    assert st["max_abs_logk"] == pytest.approx(want["max_abs_logk"], rel=1e-12)


def test_stats_sequence_operator_reading():
    """Under Seq-TIS every valid token of a response whose K exceeds C is
    flagged and carries w = C; the excess adds each such token's own ratio
    minus C.  One response with k = 2, 1.5, 1 (K = 3 > 2) and one with
    k = 1.2, 0.5 (K = 0.6)."""
    z, ids, lq, _ = _two_logit_batch([2.0, 1.5, 1.0, 1.2, 0.5])
    cu = np.array([0, 3, 5], np.int32)
    out = oracle.loss_fwd_bwd(z, ids, lq, np.ones(5), oracle.params(mode=oracle.MODE_SEQ_TIS),
                              cu_seqlens=cu, want_dz=False)
    st = out["stats"]
    assert out["trunc"].tolist() == [1, 1, 1, 0, 0]
    assert st["n_truncated"] == 3
    assert st["trunc_excess"] == pytest.approx((2 - 2) + (1.5 - 2) + (1 - 2), rel=1e-12)
    assert st["max_abs_logk"] == pytest.approx(math.log(2.0), rel=1e-12)


def _fd_setup(seed, T, V):
    rng = _rng(seed)
    z = (rng.integers(-128, 128, (T, V)) / 32).astype(np.float32)  # exact fp32 +- 2^-16
    ids = rng.integers(0, V, T).astype(np.int32)
    adv = rng.standard_normal(T) * 1.5
    lp_inf = _log_softmax(z.astype(np.float64) + rng.standard_normal((T, V)) * 0.4)[np.arange(T), ids]
    return z, ids, adv, lp_inf


@pytest.mark.parametrize("V", [2, 5, 8])
@pytest.mark.parametrize("mode", [oracle.MODE_CIS, oracle.MODE_TIS, oracle.MODE_EXACT,
                                  oracle.MODE_BAND, oracle.MODE_ICEPOP, oracle.MODE_KPOP,
                                  oracle.MODE_SEQ_TIS, oracle.MODE_SEQ_MIS])
def test_gradient_matches_central_finite_differences(V, mode):
    """d loss / d z from the oracle equals central differences of its loss with
    the weight frozen (stopgrad, Algorithm 1) and log p_old fixed.  Rows cover
    the clip-inactive and clip-active branches for both signs of A, a masked
    row, and the sequence-mean normaliser."""
    T = 6
    z, ids, adv, lp_inf = _fd_setup(100 + V + 10 * mode, T, V)
    lp0, _, _ = oracle.token_logprobs(z, ids)
    adv[:4] = [1.0, 1.0, -1.0, -1.0]
    # rho = exp(l - l_old): 1.0 (inside), 1.6 (A>0 clipped), 1.6 (A<0 flows), 0.6 (A<0 clipped)
    lp_old = lp0 - np.log([1.0, 1.6, 1.6, 0.6, 1.1, 0.9])
    mask = np.ones(T, np.uint8)
    mask[5] = 0
    cu = np.array([0, 2, 6], np.int32)
    for agg in (oracle.AGG_TOKEN_MEAN, oracle.AGG_SEQ_MEAN):
        P = oracle.params(mode=mode, agg=agg)
        base = oracle.loss_fwd_bwd(z, ids, lp_inf, adv, P, lp_old=lp_old, mask=mask,
                                   cu_seqlens=cu)
        w0 = base["w"]
        h = np.float32(2.0 ** -16)
        fd = np.zeros((T, V))
        for t in range(T):
            for j in range(V):
                zp = z.copy()
                zm = z.copy()
                zp[t, j] += h
                zm[t, j] -= h
                Lp = oracle.loss_fwd_bwd(zp, ids, lp_inf, adv, P, lp_old=lp_old, mask=mask,
                                         cu_seqlens=cu, w_fixed=w0, want_dz=False)["loss"]
                Lm = oracle.loss_fwd_bwd(zm, ids, lp_inf, adv, P, lp_old=lp_old, mask=mask,
                                         cu_seqlens=cu, w_fixed=w0, want_dz=False)["loss"]
                fd[t, j] = (Lp - Lm) / (2 * float(h))
        dz = base["dz"]
        scale = np.abs(dz).max()
        assert scale > 0
        np.testing.assert_allclose(dz, fd, rtol=0, atol=1e-7 * scale)
        assert np.all(dz[1] == 0) and np.all(dz[3] == 0) and np.all(dz[5] == 0)
        for t in (0, 2):  # rows whose operator keeps a weight carry a gradient
            assert (np.abs(dz[t]).max() > 0) == (w0[t] != 0)
        assert np.abs(dz).max() > 0


def test_on_policy_gradient_equals_snapshot_gradient_at_rho_one():
    """With no l_old the update ratio is exp(l - stopgrad l) = 1; its gradient
    equals the one taken with l_old = l (rho = 1) and the weight built from l."""
    z, ids, adv, lp_inf = _fd_setup(7, 8, 33)
    lp0, _, _ = oracle.token_logprobs(z, ids)
    P = oracle.params()
    a = oracle.loss_fwd_bwd(z, ids, lp_inf, adv, P)
    b = oracle.loss_fwd_bwd(z, ids, lp_inf, adv, P, lp_old=lp0)
    np.testing.assert_allclose(a["dz"], b["dz"], rtol=1e-13, atol=1e-18)
    assert a["loss"] == pytest.approx(b["loss"], rel=1e-13)


def test_gradient_rows_sum_to_zero():
    """sum_j dz_tj = c_t (sum_j softmax_j - 1) = 0."""
    z, ids, adv, lp_inf = _fd_setup(8, 16, 500)
    out = oracle.loss_fwd_bwd(z, ids, lp_inf, adv, oracle.params())
    rs = out["dz"].sum(axis=1)
    np.testing.assert_allclose(rs, 0.0, atol=1e-15 * np.abs(out["c"]).max() * 500)


def test_row_subset_matches_full_gradient():
    z, ids, adv, lp_inf = _fd_setup(9, 10, 40)
    full = oracle.loss_fwd_bwd(z, ids, lp_inf, adv, oracle.params())
    sub = oracle.loss_fwd_bwd(z, ids, lp_inf, adv, oracle.params(), rows=[7, 2])
    np.testing.assert_array_equal(sub["dz"], full["dz"][[7, 2]])


def test_nan_ratio_propagates():
    """A NaN log-probability gives a NaN weight in every truncating mode."""
    for mode in (oracle.MODE_CIS, oracle.MODE_TIS, oracle.MODE_EXACT):
        w, tr, _, _ = oracle.weights(np.array([np.nan, -1.0]), np.array([-1.0, np.nan]),
                                     oracle.params(mode=mode))
        assert np.isnan(w).all() and not tr.any()


def test_lmhead_chain_rule_matches_finite_differences():
    """Through the LM head z = H W^T: dH = dz W and dW = dz^T H equal central
    differences of the loss in H and W (weights frozen, l_old fixed)."""
    rng = _rng(30)
    T, Hd, V = 4, 6, 7
    Hm = rng.integers(-16, 16, (T, Hd)) / 16.0
    Wm = rng.integers(-16, 16, (V, Hd)) / 16.0
    ids = rng.integers(0, V, T)
    adv = np.array([1.0, -0.7, 0.4, -1.3])
    z0 = Hm @ Wm.T
    lp0 = _log_softmax(z0)[np.arange(T), ids]
    lp_old = lp0 - np.log([1.0, 1.1, 0.95, 1.5])   # last token: A<0, rho>1 -> flows
    lp_inf = lp0 + rng.standard_normal(T) * 0.5
    P = oracle.params()
    base = oracle.lmhead_fwd_bwd(Hm, Wm, ids, lp_inf, adv, P, lp_old=lp_old)
    w0 = base["w"]
    h = 2.0 ** -20
    def loss(Hx, Wx):
        return oracle.lmhead_fwd_bwd(Hx, Wx, ids, lp_inf, adv, P, lp_old=lp_old, w_fixed=w0,
                                     want_dw=False)["loss"]
    fdH = np.zeros_like(Hm)
    for t in range(T):
        for k in range(Hd):
            a, b = Hm.copy(), Hm.copy()
            a[t, k] += h
            b[t, k] -= h
            fdH[t, k] = (loss(a, Wm) - loss(b, Wm)) / (2 * h)
    fdW = np.zeros_like(Wm)
    for v in range(V):
        for k in range(Hd):
            a, b = Wm.copy(), Wm.copy()
            a[v, k] += h
            b[v, k] -= h
            fdW[v, k] = (loss(Hm, a) - loss(Hm, b)) / (2 * h)
    scale = max(np.abs(base["dhidden"]).max(), np.abs(base["dweight"]).max())
    np.testing.assert_allclose(base["dhidden"], fdH, rtol=0, atol=1e-8 * scale)
    np.testing.assert_allclose(base["dweight"], fdW, rtol=0, atol=1e-8 * scale)



@pytest.mark.parametrize("mode", [oracle.MODE_CIS, oracle.MODE_TIS, oracle.MODE_EXACT])
def test_lmhead_token_groups_is_the_whole_batch_computation(mode):
    """The grouped LM-head oracle (tokens taken a few at a time, for batches
    whose fp64 logits do not fit in memory) gives the per-token outputs, loss,
    statistics, dH rows and dW rows of the finite-difference-pinned
    whole-batch computation: grouping rows changes no row's arithmetic."""
    rng = _rng(31)
    T, Hd, V = 37, 16, 53
    Hm = rng.standard_normal((T, Hd))
    Wm = rng.standard_normal((V, Hd)) * 0.7
    ids = rng.integers(0, V, T)
    z0 = Hm @ Wm.T
    lp0 = _log_softmax(z0)[np.arange(T), ids]
    lp_inf = lp0 + rng.standard_normal(T) * 0.8
    adv = rng.standard_normal(T)
    mask = (rng.random(T) > 0.2).astype(np.uint8)
    lp_old = lp0 - rng.normal(0.0, 0.2, T)
    P = oracle.params(mode=mode)
    for old in (None, lp_old):
        whole = oracle.lmhead_fwd_bwd(Hm, Wm, ids, lp_inf, adv, P, lp_old=old, mask=mask)
        dw_rows = np.array([0, 5, int(ids[3]), V - 1])
        grp = oracle.lmhead_token_groups(Hm, Wm, ids, lp_inf, adv, P, lp_old=old, mask=mask,
                                         dh_rows=np.arange(T), dw_rows=dw_rows, group=5)
        for k in ("lp", "lse", "w", "c", "terms"):
            np.testing.assert_allclose(grp[k], whole[k], rtol=1e-12, atol=1e-300)
        assert np.array_equal(grp["trunc"], whole["trunc"])
        assert grp["loss"] == pytest.approx(whole["loss"], rel=1e-12)
        for k in ("n_valid", "n_truncated"):
            assert grp["stats"][k] == whole["stats"][k]
        for k in ("max_abs_logk", "trunc_excess"):
            assert grp["stats"][k] == pytest.approx(whole["stats"][k], rel=1e-12, abs=1e-300)
        sc = np.abs(whole["dweight"]).max()
        np.testing.assert_allclose(grp["dhidden"], whole["dhidden"], rtol=0, atol=1e-12 * sc)
        np.testing.assert_allclose(grp["dweight"], whole["dweight"][dw_rows], rtol=0,
                                   atol=1e-12 * sc)
        np.testing.assert_allclose(grp["dweight_abs"], whole["dweight_abs"][dw_rows],
                                   rtol=1e-12)


# ---------------------------------------------- the other operators of Table 8
def _from_p_eps(p, eps):
    """log p and log q of tokens with training probability p and log-odds
    displacement eps (Lemma 3.1: logit q = logit p - eps)."""
    p = np.asarray(p, np.float64)
    lq = -np.logaddexp(0.0, -(np.log(p) - np.log1p(-p) - eps))
    return np.log(p), lq


def test_new_operator_defaults_are_the_papers():
    """Table 8 / App. D.5 hyper-parameters are the oracle's defaults."""
    P = oracle.params()
    assert [P.icepop_lo, P.icepop_hi] == GOLDEN["icepop_band"]["value"]
    assert P.kpop_phi == GOLDEN["kpop_phi"]["value"]
    assert P.seq_cap == GOLDEN["seq_tis_cap"]["value"]
    assert [P.seq_lo, P.seq_hi] == GOLDEN["seq_mis_band"]["value"]


def test_band_lifts_exactly_where_displacement_is_below_half():
    """Two-sided band (Sec. 4.3): the lower bound (1 + p)/2 is the image of
    e^eps = 1/2 under k = p + (1 - p) e^eps, so a token is lifted iff
    e^eps < 1/2; everywhere else the band weight is the CIS weight."""
    half = GOLDEN["band_lower_displacement"]["value"]
    rng = _rng(41)
    p = rng.uniform(0.01, 0.99, 4000)
    eps = rng.uniform(-3.0, 3.0, 4000)
    eps[np.abs(eps - math.log(half)) < 1e-6] += 1e-3  # keep clear of the boundary
    lw, lq = _from_p_eps(p, eps)
    wb, trb, _, _ = oracle.weights(lw, lq, oracle.params(mode=oracle.MODE_BAND))
    wc, trc, _, _ = oracle.weights(lw, lq, oracle.params(mode=oracle.MODE_CIS))
    lifted = np.exp(eps) < half
    np.testing.assert_allclose(wb[lifted], (1.0 + p[lifted]) / 2.0, rtol=1e-14)
    assert np.all(wb[~lifted] == wc[~lifted])
    assert np.all(trb == (trc.astype(bool) | lifted))
    assert np.all(wb >= (1.0 + p) / 2.0 * (1 - 1e-15))
    # on the boundary e^eps = 1/2 exactly: k = (1 + p)/2, not lifted (the min ties)
    lw1, lq1 = _from_p_eps([0.3], [math.log(half)])
    w1, _, lk1, _ = oracle.weights(lw1, lq1, oracle.params(mode=oracle.MODE_BAND))
    assert math.exp(lk1[0]) == pytest.approx(0.65, rel=1e-14)
    assert w1[0] == pytest.approx(0.65, rel=1e-14)


def test_icepop_keeps_k_inside_its_band_and_masks_outside():
    """IcePop (Table 8): k on [0.5, 5] (bounds included), 0 outside; with a
    band wide enough to hold every ratio it is the unclamped exact ratio."""
    lo, hi = GOLDEN["icepop_band"]["value"]
    rng = _rng(42)
    lw = np.log(rng.uniform(0.01, 1.0, 3000))
    linf = lw - rng.uniform(-3.0, 3.0, 3000)
    k = np.exp(lw - linf)
    w, tr, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_ICEPOP))
    inside = (k >= lo * (1 + 1e-12)) & (k <= hi * (1 - 1e-12))
    outside = (k < lo * (1 - 1e-12)) | (k > hi * (1 + 1e-12))
    np.testing.assert_allclose(w[inside], k[inside], rtol=1e-14)
    assert np.all(w[outside] == 0.0) and np.all(tr[outside] == 1) and np.all(tr[inside] == 0)
    # exactly on the bounds: kept
    wb, trb, _, _ = oracle.weights(np.array([math.log(0.5), 0.0]),
                                   np.array([0.0, -math.log(5.0)]),
                                   oracle.params(mode=oracle.MODE_ICEPOP))
    assert trb.tolist() == [0, 0] and wb[0] == pytest.approx(0.5) and wb[1] == pytest.approx(5.0)
    wide, _, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_ICEPOP,
                                                           icepop_lo=1e-300, icepop_hi=1e300))
    np.testing.assert_allclose(wide, k, rtol=1e-14)


def test_kpop_mask_matches_binary_kl_from_library_entropy():
    """KPop-dagger (Table 8, App. D.5): the binary KL both ways, recomputed with
    scipy's relative entropy on the clamped probabilities; masked iff the
    larger exceeds phi = 2 (decided away from the threshold)."""
    special = pytest.importorskip("scipy.special")
    lo, hi = GOLDEN["kpop_clamp"]["value"]
    phi = GOLDEN["kpop_phi"]["value"]
    rng = _rng(43)
    n = 4000
    lw = np.log(rng.uniform(1e-4, 1.0, n))
    linf = np.log(rng.uniform(1e-4, 1.0, n))
    w, tr, lk, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_KPOP))
    p = np.clip(np.exp(lw), lo, hi)
    q = np.clip(np.exp(linf), lo, hi)
    kl = lambda a, b: special.rel_entr(a, b) + special.rel_entr(1 - a, 1 - b)  # noqa: E731
    m = np.maximum(kl(p, q), kl(q, p))
    clear = np.abs(m - phi) > 1e-9
    assert np.all((tr == 1)[clear] == (m > phi)[clear])
    assert np.all(w[tr == 1] == 0.0)
    keep = tr == 0
    np.testing.assert_allclose(w[keep], np.exp(lk[keep]), rtol=1e-15)
    assert 0 < tr.sum() < n
    # saturation (App. D.5): probability one on both engines is kept (metric 0
    # after the representable clamp); one on one engine only is masked when the
    # other is far from it (q = 0.5: KL(q||p) = 0.5 log(0.5 / 1e-8) + ... > 2),
    # kept when it is close (q = 0.999: about 0.012)
    w2, tr2, _, _ = oracle.weights(np.array([0.0, 0.0, 0.0]),
                                   np.array([0.0, math.log(0.5), math.log(0.999)]),
                                   oracle.params(mode=oracle.MODE_KPOP))
    assert tr2.tolist() == [0, 1, 0]
    assert w2[0] == 1.0 and w2[1] == 0.0 and w2[2] == pytest.approx(1 / 0.999)


def test_sequence_operators_use_the_product_over_each_response():
    """Seq-TIS min(K, C) and Seq-MIS K 1{K in [0.5, 2]} (Table 8), K the
    product of k over the valid tokens of a response: checked against the
    product of the per-token ratios; masked tokens are left out of K and get
    weight 0, and a token outside every response gets 0."""
    rng = _rng(44)
    T = 40
    lw = np.log(rng.uniform(0.05, 1.0, T))
    linf = lw - rng.normal(0.0, 0.3, T)
    mask = np.ones(T, np.uint8)
    mask[[3, 17, 30]] = 0
    cu = np.array([0, 1, 6, 18, 25, 37], np.int32)  # tokens 37..39 in no response
    k = np.exp(lw - linf)
    C = GOLDEN["seq_tis_cap"]["value"]
    lo, hi = GOLDEN["seq_mis_band"]["value"]
    wt, trt, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_SEQ_TIS), mask=mask,
                                   cu_seqlens=cu)
    wm, trm, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_SEQ_MIS), mask=mask,
                                   cu_seqlens=cu)
    for i in range(len(cu) - 1):
        sl = slice(cu[i], cu[i + 1])
        v = mask[sl] == 1
        K = float(np.prod(k[sl][v]))
        assert np.allclose(wt[sl][v], min(K, C), rtol=1e-12)
        assert np.all(trt[sl][v] == (K > C))
        kept = lo <= K <= hi
        assert np.allclose(wm[sl][v], K if kept else 0.0, rtol=1e-12)
        assert np.all(trm[sl][v] == (not kept))
        assert np.all(wt[sl][~v] == 0) and np.all(wm[sl][~v] == 0)
    assert np.all(wt[37:] == 0) and np.all(wm[37:] == 0)
    with pytest.raises(ValueError):
        oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_SEQ_TIS))


def test_sequence_operators_on_one_token_responses_are_token_operators():
    """With every response one token long, Seq-TIS is TIS with the same C and
    Seq-MIS is IcePop with the same band."""
    rng = _rng(45)
    T = 500
    lw = np.log(rng.uniform(0.01, 1.0, T))
    linf = lw - rng.normal(0.0, 1.0, T)
    cu = np.arange(T + 1, dtype=np.int32)
    ws, trs, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_SEQ_TIS),
                                   cu_seqlens=cu)
    wt, trt, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_TIS))
    np.testing.assert_allclose(ws, wt, rtol=1e-15)
    assert np.all(trs == trt)
    wm, trm, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_SEQ_MIS),
                                   cu_seqlens=cu)
    wi, tri, _, _ = oracle.weights(lw, linf, oracle.params(mode=oracle.MODE_ICEPOP,
                                                           icepop_lo=0.5, icepop_hi=2.0))
    np.testing.assert_allclose(wm, wi, rtol=1e-15)
    assert np.all(trm == tri)


# ---------------------------------------------------------------- entropy
def test_entropy_closed_forms():
    """Uniform rows give log V, one-hot rows 0, two-point rows the binary
    entropy; every row lies in [0, log V]; masked rows give 0."""
    V = 7
    z = np.zeros((4, V))
    z[1, 1:] = -np.inf                     # one-hot
    z[2, 2:] = -np.inf                     # two-point, p = 1/(1 + e^-1.5)
    z[2, 1] = -1.5
    z[3] = np.random.default_rng(7).standard_normal(V) * 3
    h = oracle.token_entropy(z, mask=np.array([1, 1, 1, 1], np.uint8))
    assert h[0] == pytest.approx(math.log(V), rel=1e-15)
    assert h[1] == 0.0
    p = 1.0 / (1.0 + math.exp(-1.5))
    assert h[2] == pytest.approx(-p * math.log(p) - (1 - p) * math.log(1 - p), rel=1e-14)
    assert 0.0 < h[3] < math.log(V)
    hm = oracle.token_entropy(z, mask=np.array([1, 0, 1, 0], np.uint8))
    assert hm[1] == 0.0 and hm[3] == 0.0 and hm[0] == h[0]


@pytest.mark.parametrize("V", [2, 5, 8])
def test_entropy_matches_50_digit_brute_force_and_is_shift_invariant(V):
    rng = np.random.default_rng(50 + V)
    z = rng.standard_normal((6, V)) * 4
    h = oracle.token_entropy(z)
    mpmath.mp.dps = 50
    for t in range(6):
        zs = [mpmath.mpf(float(x)) for x in z[t]]
        S = mpmath.fsum(mpmath.exp(x) for x in zs)
        ref = -mpmath.fsum((mpmath.exp(x) / S) * (x - mpmath.log(S)) for x in zs)
        assert abs(h[t] - float(ref)) <= 1e-14 * max(1.0, float(ref))
    h2 = oracle.token_entropy(z + 123.25)
    np.testing.assert_allclose(h2, h, rtol=1e-12, atol=1e-13)


# ------------------------------------------------------- mismatch diagnostics
def _softmax64(z):
    z = np.asarray(z, np.float64)
    e = np.exp(z - z.max(axis=1, keepdims=True))
    return e / e.sum(axis=1, keepdims=True)


def _diag_inputs(seed, T=5, V=9, sd=0.4):
    rng = np.random.default_rng(seed)
    z = rng.standard_normal((T, V)) * 2.0
    zi = z + rng.standard_normal((T, V)) * sd
    ids = rng.integers(0, V, T).astype(np.int32)
    return z, zi, ids


@pytest.mark.parametrize("mode", [oracle.MODE_CIS, oracle.MODE_TIS, oracle.MODE_EXACT,
                                  oracle.MODE_NONE, oracle.MODE_BAND, oracle.MODE_ICEPOP,
                                  oracle.MODE_KPOP])
def test_diagnostics_vanish_when_engines_agree(mode):
    """Identical logits: eps = log k = 0, and every operator has f(1) = 1, so
    the bias and the variance increase are 0."""
    z, _, ids = _diag_inputs(60)
    d = oracle.mismatch_diagnostics(z, z, ids, oracle.params(mode=mode))
    for k in ("eps", "logk", "bias2", "dvar"):
        assert np.all(np.abs(d[k]) < 1e-13), k


def test_diagnostics_eps_is_the_log_odds_displacement():
    """eps from Lemma 3.1's w_j definition in the normalised gauge equals
    logit p - logit q (App. A.5) and satisfies k = p + (1 - p) e^eps."""
    z, zi, ids = _diag_inputs(61, T=8)
    d = oracle.mismatch_diagnostics(z, zi, ids, oracle.params())
    p = _softmax64(z)[np.arange(8), ids]
    q = _softmax64(zi)[np.arange(8), ids]
    np.testing.assert_allclose(d["eps"], np.log(p / (1 - p)) - np.log(q / (1 - q)), atol=1e-12)
    np.testing.assert_allclose(np.exp(d["logk"]), p + (1 - p) * np.exp(d["eps"]), rtol=1e-12)
    np.testing.assert_allclose(d["p"], p, rtol=1e-13)


def test_diagnostics_closed_forms_for_no_correction_and_exact_ratio():
    """E_q[k grad log p] = sum_y p_y (e_y - p) = 0, so with no correction the
    bias vector is E_q[grad log p] = q - p and the variance is unchanged;
    the exact ratio (clamp inactive) is unbiased (Sec. 4.3) and its variance
    increase is sum_y (p_y^2 / q_y)(1 - 2 p_y + |p|^2) - (1 - |q|^2)."""
    z, zi, ids = _diag_inputs(62, T=6, V=11)
    P_, Q_ = _softmax64(z), _softmax64(zi)
    none = oracle.mismatch_diagnostics(z, zi, ids, oracle.params(mode=oracle.MODE_NONE))
    np.testing.assert_allclose(none["bias2"], ((Q_ - P_) ** 2).sum(axis=1), rtol=1e-11)
    assert np.all(np.abs(none["dvar"]) < 1e-13)
    ex = oracle.mismatch_diagnostics(z, zi, ids, oracle.params(mode=oracle.MODE_EXACT))
    assert np.all(ex["bias2"] < 1e-26)
    p2 = (P_ ** 2).sum(axis=1, keepdims=True)
    dv = ((P_ ** 2 / Q_) * (1 - 2 * P_ + p2)).sum(axis=1) - (1 - (Q_ ** 2).sum(axis=1))
    np.testing.assert_allclose(ex["dvar"], dv, rtol=1e-10)
    # a truncating operator is biased and adds less variance than the exact ratio
    cis = oracle.mismatch_diagnostics(z, zi, ids, oracle.params(mode=oracle.MODE_CIS, lam=0.2))
    assert np.all(cis["bias2"] >= 0) and np.all(cis["dvar"] <= ex["dvar"] + 1e-15)


# ---------------------------------------------------------------- confidence bins
def test_binned_sums_match_numpy_histogram():
    """Counts and per-bin sums (Sec. 4.3, Fig. 5b; App. A.5's logarithmic bins
    of 1 - p) equal numpy's histogram with the same edges: half-open bins,
    the last closed on the right, values outside the edges dropped; NaN keys
    and masked tokens are in no bin."""
    rng = _rng(71)
    T = 5000
    key = rng.uniform(-0.1, 1.1, T).astype(np.float32)
    key[::97] = np.nan
    # edges that float32 keys can equal exactly
    edges = np.array([0.0, 0.05, 0.2, 0.3, 0.5, 0.565, 0.9, 0.99, 1.0], np.float32).astype(np.float64)
    key[:8] = edges[:8]            # keys on interior edges go to the upper bin
    key[8] = 1.0                   # the last edge closes the last bin
    mask = (rng.random(T) < 0.8).astype(np.uint8)
    v1 = rng.standard_normal(T).astype(np.float32)
    v2 = rng.exponential(2.0, T).astype(np.float32)
    counts, sums = oracle.binned_sums(key, edges, [v1, v2], mask=mask)
    keep = (mask != 0) & ~np.isnan(key)
    k64 = key[keep].astype(np.float64)
    ref_c, _ = np.histogram(k64, bins=edges)
    assert np.array_equal(counts, ref_c)
    for i, v in enumerate((v1, v2)):
        ref_s, _ = np.histogram(k64, bins=edges, weights=v[keep].astype(np.float64))
        np.testing.assert_allclose(sums[i], ref_s, rtol=1e-12, atol=1e-12)
    # brute force for the edge tokens themselves
    for b in range(8):
        if mask[b]:
            assert edges[b] <= key[b] < edges[b + 1]


def test_binned_sums_of_k_minus_f_on_the_token_pass():
    """Fig. 5b's quantity: binning the sampled tokens by p and summing k - f
    gives, for CIS, zero in every bin whose tokens are all under their caps
    and the token pass's truncated excess (Lemma B.2's k - f) over all bins."""
    rng = _rng(72)
    T = 400
    lp = np.log(rng.uniform(1e-4, 0.9999, T))
    lp_inf = lp - rng.normal(0.0, 0.6, T)
    P = oracle.params(mode=oracle.MODE_CIS, lam=2.3)
    w, tr, lk, _ = oracle.weights(lp, lp_inf, P)
    k = np.exp(lk)
    edges = np.array([0.0, 0.1, 0.3, 0.565, 0.9, 0.99, 1.0])
    counts, sums = oracle.binned_sums(np.exp(lp).astype(np.float32), edges,
                                      [(k - w).astype(np.float32)])
    assert counts.sum() == T
    pbin = np.searchsorted(edges, np.exp(lp).astype(np.float32).astype(np.float64),
                           side="right") - 1
    for b in range(len(edges) - 1):
        sel = pbin == b
        if not tr[sel].any():
            assert sums[0, b] == 0.0
    excess = float(((k - w) * (tr != 0)).sum())
    np.testing.assert_allclose(sums[0].sum(), excess, rtol=1e-6)
