"""GPU parity of the mismatch diagnostics (App. A.5; Sec. 4.3, Fig. 5c-d)
against the fp64 oracle, and at full vocabulary size against closed forms.

Both kernels are covered: the streaming kernel (bf16 rows with V a multiple
of 8; CIS_DIAG_SLOT_GROUPS shrinks its ring slots so that short rows still
span many slots, wrap the ring and end in a partial slot) and the one-CTA
kernel (fp32 or ragged rows, or bf16 with CIS_DIAG_KERNEL=row).

Tolerances, from the arithmetic: eps and log k come from fp32 row sums (as log
p does in the token pass: 2e-5 plus 4 ulps).  The bias and the variance
increase are fp64 combinations of nine sums over the V candidates (P2, R2, RP,
C1 .. C5, QP: see the kernel), each of fp32 terms summed in fp32 by every
thread over its n_t candidates, then in fp64.  So each sum S carries
  |dS| <= e_c sum_j dterm_j + (n_t + 8) 2^-24 sum_j |term_j|,
where e_c = (64 + n_t) 2^-24 is one candidate's relative error (its exponent's
rounding for |exponent| <= 60 -- candidates further out weigh less than 2^-60
-- and the row's fp32 normaliser) and dterm_j bounds a term's error in units
of e_c (p, q: 1; k = p/q and a weight formed from it: 2, a weight that is a
constant of the operator: 0; a product adds its factors'; q f - p has no
cancellation bound, so it gets q f + q df + p, and its square also the
second-order e_c dr^2).  The bias and variance bounds
follow by propagating these through their closed forms to first order (plus
the second-order products) with a 25% margin, plus the fp32 rounding of the
output.  Operators whose weight jumps (IcePop, KPop) also allow each
candidate within 4 e_c of a jump to take either side.  diag_error_bounds()
computes the bound per row from fp64 softmaxes and the oracle's weights.
"""
import numpy as np
import pytest
import torch

import oracle
from _util import logits_for_oracle
from paper_2609_32444_gb300 import binding, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = torch.device("cuda")
OMODE = {"cis": oracle.MODE_CIS, "tis": oracle.MODE_TIS, "exact": oracle.MODE_EXACT,
         "none": oracle.MODE_NONE, "band": oracle.MODE_BAND, "icepop": oracle.MODE_ICEPOP,
         "kpop": oracle.MODE_KPOP}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def _rows(seed, T, V, dtype, sd=0.3):
    g = torch.Generator().manual_seed(seed)
    z = torch.randn((T, V), generator=g) * 2.5
    zi = z + torch.randn((T, V), generator=g) * sd
    ids = torch.randint(0, V, (T,), generator=g).int()
    return z.to(dtype), zi.to(dtype), ids


U = 2.0 ** -24


def n_thread(V, slot_groups=2048, threads=512):
    """Most candidates one thread sums in a row: the streaming kernel's ring
    slots of `slot_groups` groups of 8 (each of `threads` threads takes
    ceil(slot_groups / threads) groups of a slot; the defaults are its layout
    of 16 consumer warps); this also bounds the one-CTA kernel's 512 threads
    with 8-wide loads."""
    groups = -(-V // 8)
    slots = -(-groups // slot_groups)
    return 8 * slots * max(1, -(-slot_groups // threads)) + 8


def diag_error_bounds(z, zi, mode, n_t, lam=2.3, kpop_phi=2.0):
    """Per-row bounds on |kernel - exact| for bias2 and dvar (module docstring)."""
    lp = torch.log_softmax(z.double().cpu(), dim=1).numpy()
    lq = torch.log_softmax(zi.double().cpu(), dim=1).numpy()
    p, q = np.exp(lp), np.exp(lq)
    Po = oracle.params(mode=OMODE[mode], lam=lam, kpop_phi=kpop_phi)
    with np.errstate(all="ignore"):
        f = oracle.weights(lp.ravel(), lq.ravel(), Po)[0].reshape(p.shape)
        f = np.where(q > 0, f, 1.0)  # a candidate never drawn: weight irrelevant
        e_c = (64 + n_t) * U
        gam = (n_t + 8) * U
        # a weight that is a constant of the operator (no correction, a cap, a
        # clamp bound, a mask) carries no error; one formed from k = p/q does
        if mode == "none":
            df = 0 * f
        elif mode == "tis":
            df = np.where(f < 2.0, 2 * f, 0.0)
        elif mode == "exact":
            df = np.where((f > 1e-6) & (f < 1e6), 2 * f, 0.0)
        else:
            df = 2 * f
        r = q * f - p
        dr = q * f + q * df + p
        t1, t2 = q * (f * f - 1), q * (f - 1)
        d1 = q * (2 * f * df + np.abs(f * f - 1))
        d2 = q * (df + np.abs(f - 1))
        terms = {"P2": (p * p, 2 * p * p),
                 "R2": (r * r, 2 * np.abs(r) * dr + e_c * dr * dr),
                 "RP": (r * p, dr * p + np.abs(r) * p),
                 "C1": (t1 * (1 - 2 * p), d1 * np.abs(1 - 2 * p) + 2 * np.abs(t1) * p),
                 "C2": (t1, d1),
                 "C3": (t2, d2),
                 "C4": (t1 * q, d1 * q + np.abs(t1) * q),
                 "C5": (t2 * p, d2 * p + np.abs(t2) * p),
                 "QP": (q * p, 2 * q * p)}
        jump = np.zeros(p.shape, bool)
        lk = lp - lq
        if mode == "icepop":
            jump = np.minimum(np.abs(lk - np.log(0.5)), np.abs(lk - np.log(5.0))) < 4 * e_c
        elif mode == "kpop":
            lo, hi = 1e-8, 1 - 1e-8
            pc, qc = np.clip(p, lo, hi), np.clip(q, lo, hi)
            kl = np.maximum(pc * np.log(pc / qc) + (1 - pc) * np.log((1 - pc) / (1 - qc)),
                            qc * np.log(qc / pc) + (1 - qc) * np.log((1 - qc) / (1 - pc)))
            jump = np.abs(kl - kpop_phi) < 1e-4
        S, dS = {}, {}
        for k, (v, dv) in terms.items():
            S[k] = np.nansum(v, axis=1)
            dS[k] = e_c * np.nansum(dv, axis=1) + gam * np.nansum(np.abs(v), axis=1)
        if jump.any():  # either side of a jump: the term with f and with f = 0
            f0 = np.where(jump, 0.0, f)
            r0 = q * f0 - p
            alt = {"P2": 0 * p, "R2": r0 * r0 - r * r, "RP": (r0 - r) * p,
                   "C1": q * (f0 * f0 - f * f) * (1 - 2 * p), "C2": q * (f0 * f0 - f * f),
                   "C3": q * (f0 - f), "C4": q * q * (f0 * f0 - f * f), "C5": q * (f0 - f) * p,
                   "QP": 0 * p}
            for k in dS:
                dS[k] = dS[k] + np.nansum(np.abs(np.where(jump, alt[k], 0.0)), axis=1)
    C3, RP, P2, C2, C5, QP = (S[k] for k in ("C3", "RP", "P2", "C2", "C5", "QP"))
    b2 = (dS["R2"] + 2 * np.abs(C3) * dS["RP"] + np.abs(2 * RP - 2 * C3 * P2) * dS["C3"]
          + C3 ** 2 * dS["P2"] + P2 * dS["C3"] ** 2 + 2 * dS["C3"] * dS["RP"]
          + (2 * np.abs(C3) + dS["C3"]) * dS["C3"] * dS["P2"])
    dv = (dS["C1"] + P2 * dS["C2"] + np.abs(C2 - C3 * (2 + C3)) * dS["P2"] + dS["C4"]
          + np.abs(2 + 2 * C3) * dS["C5"]
          + np.abs(2 * C5 + 2 * QP - 2 * P2 - 2 * C3 * P2) * dS["C3"] + 2 * np.abs(C3) * dS["QP"]
          + dS["P2"] * dS["C2"] + dS["C3"] * (2 * dS["C5"] + 2 * dS["QP"]
                                              + (2 + 2 * np.abs(C3) + dS["C3"]) * dS["P2"]))
    return 1.25 * b2, 1.25 * dv


def _compare(out, ref, z, zi, mode, n_t, mask=None, kpop_phi=2.0):
    m = np.ones(len(ref["eps"]), bool) if mask is None else mask.astype(bool)
    bounds = dict(zip(("bias2", "dvar"), diag_error_bounds(z, zi, mode, n_t,
                                                           kpop_phi=kpop_phi)))
    got = {k: v.cpu().numpy().astype(np.float64) for k, v in out.items()}
    for k in ("eps", "logk"):
        fin = np.isfinite(ref[k][m])
        assert np.array_equal(got[k][m][~fin], ref[k][m][~fin]), k  # equal infinities
        tol = 2e-5 + 2.0 ** -21 * np.abs(ref[k][m][fin])
        assert np.all(np.abs(got[k][m][fin] - ref[k][m][fin]) <= tol), k
    assert np.all(np.abs(got["p"][m] - ref["p"][m]) <= 1e-5 * ref["p"][m] + 1e-30)
    for k in ("bias2", "dvar"):
        err = np.abs(got[k][m] - ref[k][m])
        tol = bounds[k][m] + U * np.abs(ref[k][m]) + 1e-30
        assert np.all(err <= tol), f"{k}: worst excess {np.max(err - tol):.2e}"
    for k in got:
        assert np.all(got[k][~m] == 0), k


@pytest.mark.parametrize("kernel", ["stream", "row"])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("mode", list(OMODE))
def test_diagnostics_match_oracle_small_rows(mode, dtype, kernel, monkeypatch):
    """T=24 rows of V=64 (and a ragged V=61 for fp32): every output, every token operator."""
    if kernel == "row":
        monkeypatch.setenv("CIS_DIAG_KERNEL", "row")
    elif dtype == torch.float32:
        pytest.skip("the streaming kernel takes bf16 rows")
    V = 61 if dtype == torch.float32 else 64
    z, zi, ids = _rows(3, 24, V, dtype)
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params(mode))
    torch.cuda.synchronize()
    ref = oracle.mismatch_diagnostics(logits_for_oracle(z), logits_for_oracle(zi), ids.numpy(),
                                      oracle.params(mode=OMODE[mode]))
    _compare(out, ref, z, zi, mode, n_thread(V))


@pytest.mark.parametrize("mode", ["cis", "tis", "exact"])
def test_diagnostics_v1024_recipe(mode):
    """The V=1024 recipe's two engines (noise 0.05 plus spikes of +4), masked rows included."""
    b = synth.make_batch(1, keep_infer=True)
    zi = b.extra["logits_infer"]
    m = b.mask.clone()
    m[::7] = 0
    out = binding.cis_mismatch_diagnostics(b.logits.to(DEV), zi.to(DEV), b.ids.to(DEV),
                                           binding.cis_default_params(mode), mask=m.to(DEV))
    torch.cuda.synchronize()
    ref = oracle.mismatch_diagnostics(b.logits.numpy(), zi.numpy(), b.ids.numpy(),
                                      oracle.params(mode=OMODE[mode]), mask=m.numpy())
    _compare(out, ref, b.logits, zi, mode, n_thread(b.V), m.numpy())


def test_diagnostics_full_vocabulary_closed_forms():
    """V=151936 (workload 6's recipe, 24 rows): eps = logit p - logit q (App. A.5),
    and with fp64 softmaxes from torch: no correction has bias ||q - p||^2 and
    no added variance; the exact ratio (clamp inactive here) is unbiased and
    adds sum_y (p_y^2/q_y)(1 - 2 p_y + |p|^2) - (1 - |q|^2)."""
    b = synth.make_batch(6, device=DEV, T=24)
    z, zi = b.logits, b.extra["logits_infer"]
    Pd = torch.softmax(z.double(), dim=1)
    Qd = torch.softmax(zi.double(), dim=1)
    y = b.ids.long()
    p = Pd[torch.arange(24), y]
    q = Qd[torch.arange(24), y]
    none = binding.cis_mismatch_diagnostics(z, zi, b.ids, binding.cis_default_params("none"))
    ex = binding.cis_mismatch_diagnostics(z, zi, b.ids, binding.cis_default_params("exact"))
    torch.cuda.synchronize()
    eps = (torch.log(p) - torch.log1p(-p)) - (torch.log(q) - torch.log1p(-q))
    assert torch.all((none["eps"].double() - eps).abs() <= 2e-5 + 2.0 ** -21 * eps.abs())
    n_t = n_thread(b.V)
    tb_none, tv_none = (torch.from_numpy(x).to(DEV) for x in diag_error_bounds(z, zi, "none", n_t))
    tb_ex, tv_ex = (torch.from_numpy(x).to(DEV) for x in diag_error_bounds(z, zi, "exact", n_t))
    b2 = ((Qd - Pd) ** 2).sum(dim=1)
    assert torch.all((none["bias2"].double() - b2).abs() <= tb_none + U * b2)
    assert torch.all(none["dvar"].double().abs() <= tv_none)
    kmax = (Pd / Qd).max().item()
    assert 1e-6 < (Pd / Qd).min().item() and kmax < 1e6  # the clamp is inactive
    assert torch.all(ex["bias2"].double() <= tb_ex)
    p2 = (Pd ** 2).sum(dim=1, keepdim=True)
    dv = ((Pd ** 2 / Qd) * (1 - 2 * Pd + p2)).sum(dim=1) - (1 - (Qd ** 2).sum(dim=1))
    assert torch.all((ex["dvar"].double() - dv).abs() <= tv_ex + U * dv.abs())
    cis = binding.cis_mismatch_diagnostics(z, zi, b.ids, binding.cis_default_params("cis"))
    torch.cuda.synchronize()
    tv_cis = torch.from_numpy(diag_error_bounds(z, zi, "cis", n_t)[1]).to(DEV)
    assert torch.all(cis["dvar"].double() <= ex["dvar"].double() + tv_cis + tv_ex)


def _oracle_rows_parallel(z, zi, ids, modes, lam=2.3, kpop_phi=2.0):
    """The O(V^2) oracle on a few rows for several operators at once: one
    host thread per (row, operator) (the oracle releases the GIL)."""
    from concurrent.futures import ThreadPoolExecutor
    zb, zib = logits_for_oracle(z), logits_for_oracle(zi)
    jobs = [(mode, t) for mode in modes for t in range(z.shape[0])]

    def run(job):
        mode, t = job
        return job, oracle.mismatch_diagnostics(zb[t:t + 1], zib[t:t + 1], ids[t:t + 1],
                                                oracle.params(mode=OMODE[mode], lam=lam,
                                                              kpop_phi=kpop_phi),
                                                nthreads=1)
    with ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        res = dict(ex.map(run, jobs))
    return {mode: {k: np.concatenate([res[(mode, t)][k] for t in range(z.shape[0])])
                   for k in ("eps", "logk", "p", "bias2", "dvar")} for mode in modes}


def test_diagnostics_full_vocabulary_truncating_operators_against_oracle():
    """V=151936 (workload 6's recipe): four rows spanning the confidence range
    (lowest, two middle and highest p* of 24 rows) through every operator that
    truncates -- CIS, TIS, the band, IcePop and KPop -- against the O(V^2)
    oracle (one host thread per row and operator; about a minute).  The
    recipe's N(0, 0.15^2) perturbation truncates no candidate of these rows,
    so the inference rows also get the heavy tail of App. A.2: the training
    engine's top token and 2000 random candidates lowered by 3 (k = e^3 > 5,
    above every cap and IcePop's band), 2000 raised by 1 (k = e^-1 < 0.5).
    KPop runs with phi = 0.1: at Table 8's phi = 2 the binary KL of a single
    candidate never reaches the threshold here, so it would mask nothing."""
    b = synth.make_batch(6, device=DEV, T=24)
    order = np.argsort(b.extra["pstar"].cpu().numpy())
    rows = torch.from_numpy(order[[0, 8, 16, 23]].copy()).to(DEV)
    z = b.logits[rows].contiguous()
    zi = b.extra["logits_infer"][rows].float()
    g = torch.Generator(device=DEV).manual_seed(606)
    for t in range(4):
        idx = torch.randperm(b.V, generator=g, device=DEV)[:4000]
        zi[t, idx[:2000]] -= 3.0
        zi[t, idx[2000:]] += 1.0
        zi[t, z[t].float().argmax()] -= 3.0
    zi = zi.to(torch.bfloat16).contiguous()
    ids = b.ids[rows].contiguous()
    modes = ["cis", "tis", "band", "icepop", "kpop"]
    phi = 0.1
    outs = {mode: binding.cis_mismatch_diagnostics(
        z, zi, ids, binding.cis_default_params(mode, kpop_phi=phi)) for mode in modes}
    torch.cuda.synchronize()
    refs = _oracle_rows_parallel(z.cpu(), zi.cpu(), ids.cpu().numpy(), modes, kpop_phi=phi)
    for mode in modes:
        _compare(outs[mode], refs[mode], z.cpu(), zi.cpu(), mode, n_thread(b.V), kpop_phi=phi)
    # every operator acts on these rows (KPop on the rows whose sampled-side
    # confidences leave room for a binary KL above phi), and they act differently
    for mode in modes:
        acts = refs[mode]["bias2"] > 0
        assert (acts.any() if mode == "kpop" else acts.all()), mode
    assert not np.allclose(refs["cis"]["bias2"], refs["tis"]["bias2"])


@pytest.mark.parametrize("mode", list(OMODE))
def test_diagnostics_stream_ragged_slots(mode, monkeypatch):
    """The streaming kernel with 64-group slots (V=2056: four full slots and a
    one-group slot per pass), sampled ids on slot edges, masked rows, and
    more rows than SMs per CTA only through the row loop (T=24)."""
    monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", "64")
    V, T = 2056, 24
    z, zi, ids = _rows(11, T, V, torch.bfloat16, sd=0.5)
    ids[:8] = torch.tensor([0, V - 1, 511, 512, 1023, 1024, 2047, 2048], dtype=torch.int32)
    m = torch.ones(T, dtype=torch.uint8)
    m[[5, 17]] = 0
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params(mode), mask=m.to(DEV))
    torch.cuda.synchronize()
    ref = oracle.mismatch_diagnostics(logits_for_oracle(z), logits_for_oracle(zi), ids.numpy(),
                                      oracle.params(mode=OMODE[mode]), mask=m.numpy())
    _compare(out, ref, z, zi, mode, n_thread(V, 64), m.numpy())


def test_diagnostics_slot_sizes_agree(monkeypatch):
    """The same bf16 rows (V=24576: 3072 groups, so every consumer warp holds
    groups in a full slot) through ring slots of 16 and 24 warps, of 8 warps
    in two CTAs per SM and 4 in four, of 64, 7 and 1 groups (the last wraps
    the ring hundreds of times per pass) and the one-CTA kernel: results
    differ by summation order only."""
    V, T = 24576, 16
    z, zi, ids = _rows(12, T, V, torch.bfloat16)
    P = binding.cis_default_params("cis")
    outs = []
    configs = [("16", None), ("24", None), ("8", None), ("4", None), ("16", "64"), ("16", "7"),
               ("24", "1")]
    # a full slot holds four groups per consumer thread
    n_ts = [n_thread(V, int(sg or 128 * int(w)), 32 * int(w)) for w, sg in configs]
    n_ts.append(n_thread(V))
    for warps, sg in configs:
        monkeypatch.setenv("CIS_DIAG_WARPS", warps)
        if sg is None:
            monkeypatch.delenv("CIS_DIAG_SLOT_GROUPS", raising=False)
        else:
            monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", sg)
        outs.append(binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV), P))
    monkeypatch.setenv("CIS_DIAG_KERNEL", "row")
    outs.append(binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV), P))
    torch.cuda.synchronize()
    # each result carries its own fp32 summation error (slots of 1 group put
    # all 24576 candidates of a row in one thread's sums): two results may
    # differ by the sum of their bounds
    bounds = [dict(zip(("bias2", "dvar"), diag_error_bounds(z, zi, "cis", n))) for n in n_ts]
    base = {k: v.double().cpu().numpy() for k, v in outs[0].items()}
    for o, bd in zip(outs[1:], bounds[1:]):
        for k, v in o.items():
            d = np.abs(v.double().cpu().numpy() - base[k])
            if k in ("bias2", "dvar"):
                tol = bounds[0][k] + bd[k] + 2 * U * np.abs(base[k])
            elif k == "p":
                tol = 2e-5 * base[k]
            else:
                tol = 2 * (2e-5 + 2.0 ** -21 * np.abs(base[k]))
            assert np.all(d <= tol), k


def test_diagnostics_many_rows_per_cta():
    """T=700 rows of V=1024 (several rows per CTA on any GPU), every fifth
    masked: each row matches the oracle."""
    V, T = 1024, 700
    z, zi, ids = _rows(14, T, V, torch.bfloat16)
    m = torch.ones(T, dtype=torch.uint8)
    m[::5] = 0
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params("cis"), mask=m.to(DEV))
    torch.cuda.synchronize()
    ref = oracle.mismatch_diagnostics(logits_for_oracle(z), logits_for_oracle(zi), ids.numpy(),
                                      oracle.params(mode=oracle.MODE_CIS), mask=m.numpy())
    _compare(out, ref, z, zi, "cis", n_thread(V), m.numpy())


def test_diagnostics_several_rows_per_cta_with_short_slots(monkeypatch):
    """T=400 rows of V=2056 through 64-group slots (five slots a pass), so
    that every CTA walks two or three rows, with every third row masked and
    two bad ids: the producer's L2 prefetch of a CTA's next valid row skips
    the masked ones, and the epilogue warp's per-row buffers alternate
    between the rows that remain.  Every row matches the oracle."""
    monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", "64")
    V, T = 2056, 400
    z, zi, ids = _rows(21, T, V, torch.bfloat16)
    m = torch.ones(T, dtype=torch.uint8)
    m[::3] = 0
    bad = [155, 307]  # valid rows (not multiples of 3) with ids out of range
    ids[bad[0]] = V
    ids[bad[1]] = -1
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params("cis"), mask=m.to(DEV),
                                           dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == binding.CIS_ERR_BAD_TOKEN_ID
    for k, v in out.items():
        assert torch.isnan(v[bad]).all(), k
    keep = m.numpy().astype(bool)
    keep[bad] = False  # compared as masked below: the oracle takes in-range ids only
    ids_ok = ids.clone()
    ids_ok[bad] = 0
    ref = oracle.mismatch_diagnostics(logits_for_oracle(z), logits_for_oracle(zi), ids_ok.numpy(),
                                      oracle.params(mode=oracle.MODE_CIS), mask=keep.astype(np.uint8))
    got = {k: v.clone() for k, v in out.items()}
    for k in got:
        got[k][bad] = 0.0
    _compare(got, ref, z, zi, "cis", n_thread(V, 64), keep.astype(np.uint8))


def test_diagnostics_all_other_entries_neg_inf(monkeypatch):
    """A row whose entries other than y are -inf for the training engine
    (p = 1, every other candidate has k = f = 0).  logit p is infinite there:
    eps is not finite on either side (the kernel's log-odds give +inf, the
    oracle's definition NaN); the other outputs agree."""
    monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", "64")
    V, T = 2056, 4
    z, zi, ids = _rows(13, T, V, torch.bfloat16)
    z[0, :] = float("-inf")
    z[0, ids[0]] = 1.0
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params("cis"))
    torch.cuda.synchronize()
    ref = oracle.mismatch_diagnostics(logits_for_oracle(z), logits_for_oracle(zi), ids.numpy(),
                                      oracle.params(mode=oracle.MODE_CIS))
    assert not np.isfinite(out["eps"][0].item()) and not np.isfinite(ref["eps"][0])
    assert out["p"][0].item() == 1.0
    out["eps"][0] = 0.0
    ref["eps"][0] = 0.0
    _compare(out, ref, z, zi, "cis", n_thread(V, 64))


@pytest.mark.parametrize("kernel", ["stream", "row"])
def test_diagnostics_huge_magnitude_logits(kernel, monkeypatch):
    """Rows at near-zero temperature: logits of magnitude ~1e4 in bf16, so a
    thread's first groups can all lie thousands below zero (a running sum
    started there must stay 0, not 0 x inf), with ties at the top and the
    sampled token among them in some rows."""
    if kernel == "row":
        monkeypatch.setenv("CIS_DIAG_KERNEL", "row")
    monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", "64")
    V, T = 4096, 12
    g = torch.Generator().manual_seed(21)
    z = (torch.randn((T, V), generator=g) * 4e3).to(torch.bfloat16)
    ids = torch.randint(0, V, (T,), generator=g).int()
    top = z.float().argmax(dim=1)
    for t in range(0, T, 2):  # a tie at the top, y one of the two
        z[t, (top[t] + 1) % V] = z[t, top[t]]
        ids[t] = top[t]
    zi = z.clone()
    zi[1::2] = (z[1::2].float() + torch.randn((T // 2, V), generator=g) * 300.0).to(torch.bfloat16)
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params("cis"))
    torch.cuda.synchronize()
    ref = oracle.mismatch_diagnostics(logits_for_oracle(z), logits_for_oracle(zi), ids.numpy(),
                                      oracle.params(mode=oracle.MODE_CIS))
    for k in out:
        assert not torch.isnan(out[k]).any(), k
    # rows with p = 1 exactly have an infinite (kernel) or undefined (oracle) eps
    fin = np.isfinite(ref["eps"])
    sel = torch.from_numpy(fin).to(DEV)
    _compare({k: v[sel] for k, v in out.items()}, {k: v[fin] for k, v in ref.items()},
             z[torch.from_numpy(fin)], zi[torch.from_numpy(fin)], "cis", n_thread(V, 64))


def test_diagnostics_full_vocabulary_low_temperature_rows():
    """Rows 12040, 13614, 14810 and 15007 of workload 6 as generated on the
    GPU (V=151936): near-zero temperature, a tie or a single token at the top
    (p = 0.5 or ~1) and logits far below it.  A pass-1 running sum started on
    a group thousands below zero once overflowed its rescale (0 x inf = NaN)
    here; the outputs must be finite (eps may be infinite) and match fp64
    closed forms, as in the closed-form test above."""
    b = synth.make_batch(6, device=DEV, T=16384)
    rows = torch.tensor([12040, 13614, 14810, 15007], device=DEV)
    z, zi = b.logits[rows].contiguous(), b.extra["logits_infer"][rows].contiguous()
    ids = b.ids[rows].contiguous()
    none = binding.cis_mismatch_diagnostics(z, zi, ids, binding.cis_default_params("none"))
    torch.cuda.synchronize()
    for k in none:
        assert torch.isfinite(none[k]).all() or k == "eps", (k, none[k])
    Pd = torch.softmax(z.double(), dim=1)
    Qd = torch.softmax(zi.double(), dim=1)
    p = Pd[torch.arange(4), ids.long()]
    assert torch.all((none["p"].double() - p).abs() <= 1e-5 * p + 1e-30)
    b2 = ((Qd - Pd) ** 2).sum(dim=1)
    assert torch.all((none["bias2"].double() - b2).abs() <= 1e-3 * b2 + 2e-5)
    assert torch.all(none["dvar"].double().abs() <= 2e-5)


def test_diagnostics_full_workload_every_row():
    """The benchmarked workload (T=16384, V=151936, GPU-generated) in the
    launch the benchmark times: on every row p in (0, 1], bias2 >= 0 and
    finite, dvar finite, and eps NaN-free except where p = 1; and eight
    sampled rows against the O(V^2) oracle (one host thread each, about 40 s).
    With one CTA per SM a CTA walks rows c, c + grid, ..., so the samples
    take each CTA's first and second row (both parities of the per-row
    buffers), rows deep into a CTA's sequence (the ring, the L2 prefetch of
    the next row and the epilogue warp long in steady state) and the last row
    of the batch."""
    b = synth.make_batch(6, device=DEV)
    outs = {}
    for mode in ("cis", "exact"):
        out = binding.cis_mismatch_diagnostics(b.logits, b.extra["logits_infer"], b.ids,
                                               binding.cis_default_params(mode))
        torch.cuda.synchronize()
        p = out["p"]
        assert torch.all((p > 0) & (p <= 1)), mode
        assert torch.isfinite(out["bias2"]).all() and torch.all(out["bias2"] >= -1e-6), mode
        assert torch.isfinite(out["dvar"]).all() and torch.isfinite(out["logk"]).all(), mode
        assert not torch.isnan(out["eps"][p < 1]).any(), mode
        outs[mode] = out
    grid = min(b.T, torch.cuda.get_device_properties(DEV).multi_processor_count)
    picks = [0, grid, 75 + 53 * grid, 75 + 54 * grid, 5000, 12345, b.T - 1 - grid, b.T - 1]
    rows = torch.tensor(sorted({t for t in picks if 0 <= t < b.T}), device=DEV)
    z = b.logits[rows].cpu()
    zi = b.extra["logits_infer"][rows].cpu()
    ids = b.ids[rows].cpu().numpy()
    ref = _oracle_rows_parallel(z, zi, ids, ["cis"])["cis"]
    got = {k: v[rows] for k, v in outs["cis"].items()}
    _compare(got, ref, z, zi, "cis", n_thread(b.V))


@pytest.mark.parametrize("dtype,V", [(torch.float32, 64), (torch.bfloat16, 2056)])
def test_diagnostics_bad_id_and_status(dtype, V, monkeypatch):
    monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", "64")
    z, zi, ids = _rows(4, 8, V, dtype)
    ids[3] = V
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    out = binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV),
                                           binding.cis_default_params(), dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & binding.CIS_ERR_BAD_TOKEN_ID
    assert all(torch.isnan(out[k][3]).item() for k in out)
    assert not any(torch.isnan(out[k][:3]).any().item() for k in out)
