"""GPU parity of the per-token softmax entropy (App. D's logged training-policy
entropy) against the fp64 oracle, from every entry point that can return it,
and a check that asking for it changes the other outputs by rounding at most.

Tolerance, from the arithmetic: the kernels keep s = sum e^{z - m} and
u = sum e^{z - m} (z - m) in fp32 over V terms and form
H = -p log p - (1 - p) log(1 - p) + (1 - p)(log s - u / s); each sum carries a
relative error of a few 1e-7 for the row sizes here, so |H_gpu - H| is held to
2e-5 H + 2e-6.
"""
import numpy as np
import pytest
import torch

import oracle
from _util import bf16_tensor_bits, bf16_ulp_distance, logits_for_oracle
from paper_2609_32444_gb300 import binding, synth
from test_gpu_parity import DEV, to_dev

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def _check_h(got, want, mask=None):
    got = got.cpu().numpy().astype(np.float64) if torch.is_tensor(got) else got
    assert np.array_equal(np.isnan(got), np.isnan(want))
    ok = ~np.isnan(want)
    err = np.abs(got[ok] - want[ok])
    assert np.all(err <= 2e-5 * np.abs(want[ok]) + 2e-6), f"worst {err.max():.3e}"
    if mask is not None:
        assert np.all(got[~mask.astype(bool)] == 0)


def _same_up_to_rounding(a, b, rel=2.0 ** -21, abs_=1e-7):
    """The entropy variants reduce the same sums; the compiler may still fuse
    a multiply into an add differently, so values agree to fp32 rounding."""
    x = a.double().cpu().numpy()
    y = b.double().cpu().numpy()
    assert np.array_equal(np.isnan(x), np.isnan(y))
    ok = ~np.isnan(x)
    assert np.all(np.abs(x[ok] - y[ok]) <= rel * np.abs(y[ok]) + abs_)


@pytest.mark.parametrize("cfg,T", [(1, None), (2, 512), (3, 32)])
def test_forward_entropy(cfg, T):
    """cis_token_logprobs: fp32 V=1024, bf16 V=32000 with padding, and the
    V=151936 temperature recipe (p from 1e-4 to 0.9999)."""
    b = synth.make_batch(cfg, device=DEV if cfg >= 3 else "cpu", T=T)
    g = to_dev(b)
    lp, _, h = binding.cis_token_logprobs(g["logits"], g["ids"], mask=g["mask"], want_entropy=True)
    lp_plain = binding.cis_token_logprobs(g["logits"], g["ids"], mask=g["mask"])
    torch.cuda.synchronize()
    ref = oracle.token_entropy(logits_for_oracle(b.logits), mask=b.mask.cpu().numpy())
    _check_h(h, ref, b.mask.cpu().numpy())
    _same_up_to_rounding(lp, lp_plain)


@pytest.mark.parametrize("kind", ["neg_inf", "one_hot", "flat", "ties", "huge", "nan"])
def test_entropy_edge_rows(kind):
    """-inf entries, one-hot rows (H = 0), flat rows (H = log V), ties, logits
    of magnitude ~1e4 and NaN rows, through the fused pass."""
    b = synth.make_edge_rows(kind, V=1024, T=16, dtype=torch.float32)
    g = to_dev(b)
    P = binding.cis_default_params("cis")
    out = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                   dlogits_dtype=torch.float32, want_entropy=True)
    torch.cuda.synchronize()
    ref = oracle.token_entropy(logits_for_oracle(b.logits), mask=b.mask.cpu().numpy())
    _check_h(out["entropy"], ref, b.mask.cpu().numpy())


@pytest.mark.parametrize("cfg,T,dz", [(1, None, torch.float32), (3, 48, torch.bfloat16),
                                      (2, 300, torch.bfloat16)])
def test_fused_pass_entropy_changes_nothing_else(cfg, T, dz):
    """The fused pass (row-wise kernel for V=1024 fp32 and V=32000, the cluster
    kernel for V=151936): entropy matches the oracle, stats.entropy_sum is its
    sum over valid tokens, and dlogits, lp, w, trunc and the loss equal those
    of the call without entropy up to fp32 rounding (dlogits within one step
    of its type)."""
    b = synth.make_batch(cfg, device=DEV if cfg >= 3 else "cpu", T=T)
    g = to_dev(b)
    P = binding.cis_default_params("cis", lam=b.lam)
    kw = dict(mask=g["mask"], dlogits_dtype=dz)
    a = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, **kw)
    e = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, want_entropy=True,
                                 **kw)
    torch.cuda.synchronize()
    _same_up_to_rounding(e["lp"], a["lp"])
    _same_up_to_rounding(e["w"], a["w"], rel=1e-5)  # w = e^{lp - lq}: lp's rounding, relative
    assert torch.equal(e["trunc"], a["trunc"])
    da, de = a["dlogits"], e["dlogits"]
    if dz == torch.bfloat16:
        d = bf16_ulp_distance(bf16_tensor_bits(de), bf16_tensor_bits(da))
        assert d.max() <= 1
    else:
        _same_up_to_rounding(de, da, rel=2.0 ** -20, abs_=1e-9)
    la, le = float(a["loss"].cpu()[0]), float(e["loss"].cpu()[0])
    # the loss is a cancelling sum: compare on the scale of sum_t |term_t|
    m = b.mask.cpu().numpy().astype(bool)
    terms = np.abs(a["w"].double().cpu().numpy() * b.adv.cpu().numpy())[m].sum() / max(1, m.sum())
    assert abs(la - le) <= 1e-6 * terms + 1e-15
    m = b.mask.cpu().numpy()
    ref = oracle.token_entropy(logits_for_oracle(b.logits), mask=m)
    _check_h(e["entropy"], ref, m)
    st = binding.decode_stats(e["stats"])
    assert st["entropy_sum"] == pytest.approx(float(e["entropy"].double().sum()), rel=1e-12)
    assert binding.decode_stats(a["stats"])["entropy_sum"] == 0.0


def test_host_path_entropy():
    b = synth.make_batch(1)
    P = binding.cis_default_params("cis", lam=b.lam)
    dz = torch.empty((b.T, b.V), dtype=torch.float32).pin_memory()
    out = binding.cis_loss_fwd_bwd_host(b.logits, b.ids, b.lp_infer, b.adv, P, dz, mask=b.mask,
                                        chunk_tokens=40, want_entropy=True)
    torch.cuda.synchronize()
    ref = oracle.token_entropy(b.logits.numpy(), mask=b.mask.numpy())
    _check_h(out["entropy"].numpy().astype(np.float64), ref, b.mask.numpy())


def test_lmhead_entropy():
    """The LM head: entropy from the forward sweep's tiles of H W^T."""
    b = synth.make_batch(5, T=200, V=1000, H=256)
    P = binding.cis_default_params("cis", lam=b.lam)
    out = binding.cis_lmhead_fused(b.hidden.to(DEV), b.weight.to(DEV), b.ids.to(DEV),
                                   b.lp_infer.to(DEV), b.adv.to(DEV), P, mask=b.mask.to(DEV),
                                   want_entropy=True)
    plain = binding.cis_lmhead_fused(b.hidden.to(DEV), b.weight.to(DEV), b.ids.to(DEV),
                                     b.lp_infer.to(DEV), b.adv.to(DEV), P, mask=b.mask.to(DEV))
    torch.cuda.synchronize()
    hb = b.hidden.contiguous().view(torch.int16).numpy().view(np.uint16)
    wb = b.weight.contiguous().view(torch.int16).numpy().view(np.uint16)
    Z = oracle.bf16_bits_to_f64(hb) @ oracle.bf16_bits_to_f64(wb).T
    ref = oracle.token_entropy(Z, mask=b.mask.numpy())
    _check_h(out["entropy"], ref, b.mask.numpy())
    _same_up_to_rounding(out["lp"], plain["lp"])
    _same_up_to_rounding(out["w"], plain["w"], rel=1e-5)
    for k in ("dhidden", "dweight"):  # fp32 products of dz rounded to bf16 either way
        x, y = out[k].double(), plain[k].double()
        scale = y.abs().max().item()
        assert (x - y).abs().max().item() <= 2.0 ** -8 * scale
