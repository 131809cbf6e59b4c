"""GPU parity of the token pass fused with the LM head (cis_lmhead_fused)
against the fp64 oracle (logits H W^T in fp64, the pinned token pass, and the
chain rule dH = dz W, dW = dz^T H).

Tolerances, derived from the arithmetic of the path:
  - log p, weights, truncation decisions and loss: as for the logits entry
    points (2e-5 + 4 fp32 ulps, 1e-5 relative, the 4e-5 decision band,
    1e-5 of sum |term|); the logits are fp32 sums of exact bf16 products, off
    by ~1e-6 from fp64.
  - dH and dW: dz enters the two products rounded to bf16 (relative 2^-9), and
    the products accumulate K terms in fp32 (relative K 2^-24 at worst).  So
    |dH_gpu - dH| <= (2^-8 + K 2^-24) (|dz| |W|) elementwise, with (|dz| |W|)
    from the oracle, K = V for dH and K = T for dW; a bf16 output adds 2^-8
    |dH| for its own rounding.
"""
import numpy as np
import pytest
import torch

import oracle
from _util import bf16_tensor_bits
from paper_2609_32444_gb300 import binding, synth
from test_gpu_parity import check_stats

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = torch.device("cuda")
MODE_ID = {"cis": oracle.MODE_CIS, "tis": oracle.MODE_TIS, "exact": oracle.MODE_EXACT,
           "none": oracle.MODE_NONE}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def _bits(t):
    return bf16_tensor_bits(t)


def _run(b, mode="cis", grad_dtype=torch.float32, lp_old=None, chunk=None):
    P = binding.cis_default_params(mode, lam=b.lam)
    return binding.cis_lmhead_fused(b.hidden.to(DEV), b.weight.to(DEV), b.ids.to(DEV),
                                    b.lp_infer.to(DEV), b.adv.to(DEV), P,
                                    lp_old=None if lp_old is None else lp_old.to(DEV),
                                    mask=b.mask.to(DEV), grad_dtype=grad_dtype, chunk=chunk)


def _oracle(b, mode="cis", rows=None, lp_old=None):
    m = b.mask.cpu().numpy()
    return oracle.lmhead_fwd_bwd(_bits(b.hidden), _bits(b.weight), b.ids.cpu().numpy(),
                                 b.lp_infer.cpu().numpy(), b.adv.cpu().numpy(),
                                 oracle.params(mode=MODE_ID[mode], lam=b.lam), mask=m,
                                 rows=rows, n_valid_total=int(m.sum()),
                                 lp_old=None if lp_old is None else lp_old.cpu().numpy())


def _check_tokens(out, ref, rows, b, mode, full):
    lp = out["lp"].cpu().numpy()[rows].astype(np.float64)
    w = out["w"].cpu().numpy()[rows].astype(np.float64)
    tr = out["trunc"].cpu().numpy()[rows]
    assert np.all(np.abs(lp - ref["lp"]) <= 2e-5 + 2.0 ** -21 * np.abs(ref["lp"]))
    assert np.all(np.abs(w - ref["w"]) <= 1e-5 * np.abs(ref["w"]) + 1e-30)
    li = b.lp_infer.cpu().numpy()[rows].astype(np.float64)
    logk = ref["lp"] - li
    if mode == "cis":
        cap = np.log1p(b.lam * np.maximum(-np.expm1(ref["lp"]), 5e-3))
        band = np.abs(logk - cap) < 4e-5
    else:
        band = np.zeros(len(rows), bool)
    assert not np.any((tr != ref["trunc"]) & ~band)
    if full:
        loss = float(out["loss"].cpu()[0])
        assert abs(loss - ref["loss"]) <= 1e-5 * np.abs(ref["terms"]).sum() + 1e-300
        check_stats(out["stats"], ref, li, band=band, tr_gpu=tr)


def _check_grad(got, want, want_abs, K, bf16_out):
    g = got.float().cpu().numpy().astype(np.float64)
    tol = (2.0 ** -8 + K * 2.0 ** -24) * want_abs + 1e-30
    if bf16_out:
        tol = tol + 2.0 ** -8 * np.abs(want)
    err = np.abs(g - want)
    bad = err > tol
    assert not bad.any(), f"{bad.sum()} entries off; worst excess {(err - tol).max():.3e}"


@pytest.mark.parametrize("T,V,H,grad", [(256, 1024, 256, torch.float32),
                                        (200, 1000, 512, torch.float32),
                                        (256, 1024, 256, torch.bfloat16)])
def test_lmhead_small_every_element(T, V, H, grad):
    """Every per-token output, the loss, dH and dW, including ragged token and
    vocabulary tiles (T=200, V=1000)."""
    b = synth.make_batch(5, T=T, V=V, H=H)
    out = _run(b, grad_dtype=grad)
    torch.cuda.synchronize()
    ref = _oracle(b)
    rows = np.arange(T)
    _check_tokens(out, ref, rows, b, "cis", full=True)
    _check_grad(out["dhidden"], ref["dhidden"], ref["dhidden_abs"], V, grad == torch.bfloat16)
    _check_grad(out["dweight"], ref["dweight"], ref["dweight_abs"], T, grad == torch.bfloat16)
    st = binding.decode_stats(out["stats"])
    assert st["status"] == 0 and st["n_valid"] == int(b.mask.sum())


@pytest.mark.parametrize("mode", ["cis", "tis", "exact"])
def test_lmhead_hidden_2048(mode):
    """The workload's hidden size (H=2048) on T=512, V=4096: every element."""
    b = synth.make_batch(5, T=512, V=4096)
    out = _run(b, mode)
    torch.cuda.synchronize()
    ref = _oracle(b, mode)
    _check_tokens(out, ref, np.arange(b.T), b, mode, full=True)
    _check_grad(out["dhidden"], ref["dhidden"], ref["dhidden_abs"], b.V, False)
    _check_grad(out["dweight"], ref["dweight"], ref["dweight_abs"], b.T, False)


@pytest.mark.parametrize("T,V,H,chunk,grad", [(200, 1000, 512, 256, torch.float32),
                                              (300, 4096, 2048, 1024, torch.bfloat16),
                                              (130, 2000, 256, 768, torch.float32)])
def test_lmhead_vocabulary_chunks(T, V, H, chunk, grad):
    """A workspace sized for narrow vocabulary chunks: dH accumulates over the
    chunks, dW is written chunk by chunk, the last chunk ragged; every element."""
    b = synth.make_batch(5, T=T, V=V, H=H)
    out = _run(b, grad_dtype=grad, chunk=chunk)
    torch.cuda.synchronize()
    ref = _oracle(b)
    _check_tokens(out, ref, np.arange(T), b, "cis", full=True)
    _check_grad(out["dhidden"], ref["dhidden"], ref["dhidden_abs"], V, grad == torch.bfloat16)
    _check_grad(out["dweight"], ref["dweight"], ref["dweight_abs"], T, grad == torch.bfloat16)
    assert binding.decode_stats(out["stats"])["status"] == 0


@pytest.mark.parametrize("grad", [torch.float32, torch.bfloat16])
def test_lmhead_outputs_16_byte_aligned(grad):
    """Gradient buffers that are 16-byte but not 32-byte aligned take the
    16-byte store path; the results equal those of aligned buffers bit for
    bit (the same arithmetic, only the store width differs)."""
    b = synth.make_batch(5, T=200, V=1000, H=256)
    T, H, V = 200, 256, 1000
    es = torch.empty((), dtype=grad).element_size()
    pad = 16 // es
    dh_buf = torch.empty(T * H + pad, dtype=grad, device=DEV)
    dw_buf = torch.empty(V * H + pad, dtype=grad, device=DEV)
    dh = dh_buf[pad:].view(T, H)
    dw = dw_buf[pad:].view(V, H)
    assert dh.data_ptr() % 32 == 16 and dw.data_ptr() % 32 == 16
    P = binding.cis_default_params("cis", lam=b.lam)
    args = (b.hidden.to(DEV), b.weight.to(DEV), b.ids.to(DEV), b.lp_infer.to(DEV),
            b.adv.to(DEV), P)
    kw = dict(mask=b.mask.to(DEV), grad_dtype=grad, chunk=256)
    odd = binding.cis_lmhead_fused(*args, dhidden=dh, dweight=dw, **kw)
    ref = binding.cis_lmhead_fused(*args, **kw)
    torch.cuda.synchronize()
    assert ref["dhidden"].data_ptr() % 32 == 0 and ref["dweight"].data_ptr() % 32 == 0
    assert torch.equal(odd["dhidden"].view(torch.int16 if es == 2 else torch.int32),
                       ref["dhidden"].view(torch.int16 if es == 2 else torch.int32))
    assert torch.equal(odd["dweight"].view(torch.int16 if es == 2 else torch.int32),
                       ref["dweight"].view(torch.int16 if es == 2 else torch.int32))


@pytest.mark.parametrize("T,V,H,chunk,grad", [(300, 1100, 256, 768, torch.float32),
                                              (512, 4096, 2048, None, torch.float32),
                                              (130, 1900, 512, 512, torch.bfloat16)])
def test_lmhead_multicast_clusters_bit_identical(monkeypatch, T, V, H, chunk, grad):
    """Every GEMM on 2-CTA clusters sharing each B tile (multicast, the
    default) against every GEMM on one CTA (CIS_LMHEAD_MC=0), each with a
    chunk's dH and dW in one launch (the default) and in two
    (CIS_LMHEAD_DUAL=0): the same tiles with the same MMAs and epilogues, so
    every output matches bit for bit.  T=300 gives an odd number of 128-row
    token tiles (FWD, DZ, DH), and the last chunks of 332 and 364 columns odd
    numbers of 128-column vocabulary tiles (DW), so the padding tile of the
    last pair is exercised; the first case is also checked against the
    oracle."""
    b = synth.make_batch(5, T=T, V=V, H=H)
    outs = {}
    for mc in ("15", "0"):
        for dual in ("1", "0"):
            monkeypatch.setenv("CIS_LMHEAD_MC", mc)
            monkeypatch.setenv("CIS_LMHEAD_DUAL", dual)
            outs[mc, dual] = _run(b, grad_dtype=grad, chunk=chunk)
    torch.cuda.synchronize()
    a = outs["15", "1"]
    for key, r in outs.items():
        for k in ("lp", "w", "trunc", "dhidden", "dweight", "loss"):
            x, y = a[k], r[k]
            if x.dtype.is_floating_point:
                x = x.view(torch.int16 if x.element_size() == 2 else
                           (torch.int32 if x.element_size() == 4 else torch.int64))
                y = y.view(x.dtype)
            assert torch.equal(x, y), (key, k)
        assert binding.decode_stats(r["stats"])["status"] == 0, key
    if T == 300:
        ref = _oracle(b)
        _check_tokens(a, ref, np.arange(T), b, "cis", full=True)
        _check_grad(a["dhidden"], ref["dhidden"], ref["dhidden_abs"], V, False)
        _check_grad(a["dweight"], ref["dweight"], ref["dweight_abs"], T, False)


def test_lmhead_workspace_too_small():
    """Less workspace than 256-column chunks need is refused on the host."""
    b = synth.make_batch(5, T=64, V=1024, H=256)
    need = binding.cis_lmhead_workspace_size_chunk(64, 1024, 256, 256)
    ws = torch.empty(need + 1024, dtype=torch.uint8, device=DEV)
    off = (-ws.data_ptr()) % 1024
    P = binding.cis_default_params("cis", lam=b.lam)
    with pytest.raises(RuntimeError):
        binding.cis_lmhead_fused(b.hidden.to(DEV), b.weight.to(DEV), b.ids.to(DEV),
                                 b.lp_infer.to(DEV), b.adv.to(DEV), P, mask=b.mask.to(DEV),
                                 workspace=ws[off:off + need - 4096], chunk=None)


def test_lmhead_masked_tokens_and_old_logprobs():
    """Masked tokens contribute nothing; l_old moves rho off 1 (PPO clip)."""
    b = synth.make_batch(5, T=256, V=2048, H=256)
    b.mask[::3] = 0
    base = _oracle(b)
    rng = np.random.default_rng(2)
    lp_old = torch.from_numpy((base["lp"] - rng.choice([-0.5, 0.0, 0.4], size=b.T))
                              .astype(np.float32))
    out = _run(b, lp_old=lp_old)
    torch.cuda.synchronize()
    ref = _oracle(b, lp_old=lp_old)
    _check_tokens(out, ref, np.arange(b.T), b, "cis", full=True)
    _check_grad(out["dhidden"], ref["dhidden"], ref["dhidden_abs"], b.V, False)
    _check_grad(out["dweight"], ref["dweight"], ref["dweight_abs"], b.T, False)
    m = b.mask.numpy().astype(bool)
    assert torch.count_nonzero(out["dhidden"][torch.from_numpy(~m).to(DEV)]).item() == 0


def test_lmhead_full_size_sampled_tokens():
    """T=16384, H=2048, V=151936, the benchmarked configuration and launch:
    every token's log p, w, flags, the loss and the batch statistics against
    the oracle, whose fp64 logits are formed for every token (1e13 FLOP on the
    host cores, in groups of tokens); dH on 64 sampled tokens; dW element by
    element on 256 seeded vocabulary rows, among them the edges of every
    32768-column chunk the call works in and sampled tokens' own rows; and the
    identity sum_v dW[v] = 0 over all rows."""
    b = synth.make_batch(5, device=DEV)
    out = _run(b)
    torch.cuda.synchronize()
    rng = np.random.default_rng(5)
    rows = np.unique(np.concatenate([[0, b.T - 1], rng.integers(0, b.T, 62)]))
    edges = [e + d for e in range(0, b.V + 1, 32768) for d in (-1, 0) if 0 <= e + d < b.V]
    ys = b.ids.cpu().numpy()[rows[:16]]
    vrows = np.unique(np.concatenate([edges, [b.V - 1], ys, rng.integers(0, b.V, 256)]))[:256]
    m = b.mask.cpu().numpy()
    ref = oracle.lmhead_token_groups(_bits(b.hidden), _bits(b.weight), b.ids.cpu().numpy(),
                                     b.lp_infer.cpu().numpy(), b.adv.cpu().numpy(),
                                     oracle.params(mode=MODE_ID["cis"], lam=b.lam), mask=m,
                                     dh_rows=rows, dw_rows=vrows, group=512)
    _check_tokens(out, ref, np.arange(b.T), b, "cis", full=True)
    _check_grad(out["dhidden"][torch.from_numpy(rows).to(DEV)], ref["dhidden"],
                ref["dhidden_abs"], b.V, False)
    _check_grad(out["dweight"][torch.from_numpy(vrows).to(DEV)], ref["dweight"],
                ref["dweight_abs"], b.T, False)
    # sum_v dW[v, k] = sum_t H[t, k] sum_v dz[t, v] = 0 exactly; with dz rounded to
    # bf16 (2^-9) and fp32 accumulation over T tokens the sum is bounded by
    # sum_t |H[t, k]| sum_v |dz[t, v]| (2^-9 + T 2^-24), where
    # sum_v |dz[t, v]| = 2 |c_t| (1 - p_t) and c_t = w_t A_t / n (no l_old).
    assert torch.isfinite(out["dhidden"]).all() and torch.isfinite(out["dweight"]).all()
    dw = out["dweight"].double()
    colsum = dw.sum(dim=0).abs()
    n = float(b.mask.sum())
    c = out["w"].double() * b.adv.to(DEV).double() / n
    a = 2.0 * c.abs() * (-torch.expm1(out["lp"].double()))
    bound = (b.hidden.to(DEV).double().abs().t() @ a) * (2.0 ** -9 + b.T * 2.0 ** -24) * 1.01
    assert bool((colsum <= bound + 1e-12).all())
    st = binding.decode_stats(out["stats"])
    assert st["status"] == 0 and st["n_valid"] == b.T
