"""GPU parity of the mismatch diagnostics (App. A.5; Sec. 4.3, Fig. 5c-d)
against the fp64 oracle, and at full vocabulary size against closed forms.

Both kernels are covered: the streaming kernel (bf16 rows with V a multiple
of 8; CIS_DIAG_SLOT_GROUPS shrinks its ring slots so that short rows still
span many slots, wrap the ring and end in a partial slot) and the one-CTA
kernel (fp32 or ragged rows, or bf16 with CIS_DIAG_KERNEL=row).

Tolerances, from the arithmetic: eps and log k come from fp32 row sums (as log
p does in the token pass: 2e-5 plus 4 ulps).  The bias and the variance
increase are fp64 combinations of per-candidate fp32 terms of size O(1) (the
variances themselves are at most 1), summed in fp32 per thread: their error
is absolute, about V_thread 2^-24 with V_thread = V / 512 terms per thread.
They are held to 1e-3 of their own size plus an absolute 2e-6 (small V) or
2e-5 (V = 151936).
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


def _compare(out, ref, mask=None, abs_tol=2e-6):
    m = np.ones(len(ref["eps"]), bool) if mask is None else mask.astype(bool)
    got = {k: v.cpu().numpy().astype(np.float64) for k, v in out.items()}
    for k in ("eps", "logk"):
        fin = np.isfinite(ref[k][m])
        assert np.array_equal(got[k][m][~fin], ref[k][m][~fin]), k  # equal infinities
        tol = 2e-5 + 2.0 ** -21 * np.abs(ref[k][m][fin])
        assert np.all(np.abs(got[k][m][fin] - ref[k][m][fin]) <= tol), k
    assert np.all(np.abs(got["p"][m] - ref["p"][m]) <= 1e-5 * ref["p"][m] + 1e-30)
    for k in ("bias2", "dvar"):
        err = np.abs(got[k][m] - ref[k][m])
        tol = 1e-3 * np.abs(ref[k][m]) + abs_tol
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
    _compare(out, ref)


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
    _compare(out, ref, m.numpy())


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
    b2 = ((Qd - Pd) ** 2).sum(dim=1)
    assert torch.all((none["bias2"].double() - b2).abs() <= 1e-3 * b2 + 2e-5)
    assert torch.all(none["dvar"].double().abs() <= 2e-5)
    kmax = (Pd / Qd).max().item()
    assert 1e-6 < (Pd / Qd).min().item() and kmax < 1e6  # the clamp is inactive
    assert torch.all(ex["bias2"].double() <= 2e-5)
    p2 = (Pd ** 2).sum(dim=1, keepdim=True)
    dv = ((Pd ** 2 / Qd) * (1 - 2 * Pd + p2)).sum(dim=1) - (1 - (Qd ** 2).sum(dim=1))
    assert torch.all((ex["dvar"].double() - dv).abs() <= 1e-3 * dv.abs() + 2e-5)
    cis = binding.cis_mismatch_diagnostics(z, zi, b.ids, binding.cis_default_params("cis"))
    torch.cuda.synchronize()
    assert torch.all(cis["dvar"] <= ex["dvar"] + 2e-5)


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
    _compare(out, ref, m.numpy())


def test_diagnostics_slot_sizes_agree(monkeypatch):
    """The same bf16 rows (V=24576: 3072 groups, so every consumer warp holds
    groups in a full slot) through ring slots of 16 and 24 warps, of 64, 7
    and 1 groups (the last wraps the ring hundreds of times per pass) and the
    one-CTA kernel: results differ by summation order only."""
    V, T = 24576, 16
    z, zi, ids = _rows(12, T, V, torch.bfloat16)
    P = binding.cis_default_params("cis")
    outs = []
    for warps, sg in [("16", None), ("24", None), ("16", "64"), ("16", "7"), ("24", "1")]:
        monkeypatch.setenv("CIS_DIAG_WARPS", warps)
        if sg is None:
            monkeypatch.delenv("CIS_DIAG_SLOT_GROUPS", raising=False)
        else:
            monkeypatch.setenv("CIS_DIAG_SLOT_GROUPS", sg)
        outs.append(binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV), P))
    monkeypatch.setenv("CIS_DIAG_KERNEL", "row")
    outs.append(binding.cis_mismatch_diagnostics(z.to(DEV), zi.to(DEV), ids.to(DEV), P))
    torch.cuda.synchronize()
    # each result carries the fp32 summation error that the oracle tolerance
    # allows (slots of 1 group put all 4096 candidates in one thread's sums)
    base = {k: v.double().cpu() for k, v in outs[0].items()}
    for o in outs[1:]:
        for k, v in o.items():
            d = (v.double().cpu() - base[k]).abs()
            assert torch.all(d <= 2e-3 * base[k].abs() + 4e-6), k


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
    _compare(out, ref, m.numpy())


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
    _compare(out, ref)


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
    _compare({k: v[sel] for k, v in out.items()}, {k: v[fin] for k, v in ref.items()})


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
    """The benchmarked workload (T=16384, V=151936, GPU-generated): on every
    row p in (0, 1], bias2 >= 0 and finite, dvar finite, and eps NaN-free
    except where p = 1 (the closed-form and oracle tests fix the values)."""
    b = synth.make_batch(6, device=DEV)
    for mode in ("cis", "exact"):
        out = binding.cis_mismatch_diagnostics(b.logits, b.extra["logits_infer"], b.ids,
                                               binding.cis_default_params(mode))
        torch.cuda.synchronize()
        p = out["p"]
        assert torch.all((p > 0) & (p <= 1)), mode
        assert torch.isfinite(out["bias2"]).all() and torch.all(out["bias2"] >= -1e-6), mode
        assert torch.isfinite(out["dvar"]).all() and torch.isfinite(out["logk"]).all(), mode
        assert not torch.isnan(out["eps"][p < 1]).any(), mode


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
