"""cis_loss_fwd_bwd_noalloc: the fused pass for callers that cannot allocate
device memory -- extensions running inside a framework that owns every byte of
device memory and hands them no allocator, and C callers without one.  It takes
its scratch from a fixed array in the library's static device memory instead of
a caller workspace.

The two entry points run the same kernels on the same inputs, only with the
scratch in a different place, so every output must be bit-identical to
cis_loss_fwd_bwd's: dlogits, log p, w, the flags, the loss and the batch
statistics.  Checked through the C ABI on two calls in a row (the second call
reuses the array the first one left behind), at the largest T the array holds,
and with a sequence operator.  This file is collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_32444_gb300 import binding, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

MAX_TOKENS = 65536  # CIS_NOALLOC_MAX_TOKENS in include/cis.h


@pytest.fixture(scope="module")
def noalloc():
    from paper_2609_32444_gb300 import build
    build.build()
    L = binding.lib()
    P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    f = L.cis_loss_fwd_bwd_noalloc
    f.argtypes = [P, i32, i64, i64, i64, P, P, P, P, P, P, i64,
                  ctypes.POINTER(binding.cis_params_t), P, i32, i64, P, P, P, P, P, P, P]
    f.restype = ctypes.c_int
    return f


def _call(f, g, P, T, V, dt=torch.bfloat16, cu=None, B=0):
    dev = g["logits"].device
    out = {"dz": torch.full((T, V), float("nan"), dtype=dt, device=dev),
           "lp": torch.full((T,), float("nan"), device=dev),
           "w": torch.full((T,), float("nan"), device=dev),
           "trunc": torch.full((T,), 7, dtype=torch.uint8, device=dev),
           "stats": torch.zeros(ctypes.sizeof(binding.cis_stats_t), dtype=torch.uint8,
                                device=dev),
           "loss": torch.full((1,), float("nan"), dtype=torch.float64, device=dev)}
    ptr = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    code = binding.CIS_BF16 if dt == torch.bfloat16 else binding.CIS_F32
    in_code = binding.CIS_BF16 if g["logits"].dtype == torch.bfloat16 else binding.CIS_F32
    rc = f(ptr(g["logits"]), in_code, T, V, V, ptr(g["ids"]), ptr(g["lp"]), None,
           ptr(g["adv"]), ptr(g["mask"]), None if cu is None else ptr(cu), B, ctypes.byref(P),
           ptr(out["dz"]), code, V, ptr(out["lp"]), ptr(out["w"]), ptr(out["trunc"]), None,
           ptr(out["stats"]), ptr(out["loss"]),
           ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return rc, out


def _same(out, ref):
    """Bit-identical outputs (NaN patterns included)."""
    assert torch.equal(out["dz"].view(torch.int16 if out["dz"].element_size() == 2
                                      else torch.int32),
                       ref["dlogits"].view(torch.int16 if ref["dlogits"].element_size() == 2
                                           else torch.int32))
    assert torch.equal(out["lp"].view(torch.int32), ref["lp"].view(torch.int32))
    assert torch.equal(out["w"].view(torch.int32), ref["w"].view(torch.int32))
    assert torch.equal(out["trunc"], ref["trunc"])
    assert torch.equal(out["loss"].view(torch.int64), ref["loss"].view(torch.int64))
    assert torch.equal(out["stats"], ref["stats"])


def _dev(b):
    return {k: v.cuda() for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv,
                                         mask=b.mask, cu=b.cu_seqlens).items()}


def test_noalloc_matches_workspace_entry_point_on_two_calls(noalloc):
    b = synth.make_batch(2, T=1024, V=32000)
    g = _dev(b)
    P = binding.cis_default_params("cis", lam=b.lam)
    ref = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"])
    torch.cuda.synchronize()
    for _ in range(2):
        rc, out = _call(noalloc, g, P, b.T, b.V)
        assert rc == binding.CIS_OK
        torch.cuda.synchronize()
        st = binding.decode_stats(out["stats"])
        assert st["status"] == 0 and st["n_valid"] == int(b.mask.sum())
        _same(out, ref)


def test_noalloc_at_its_largest_token_count(noalloc):
    """T = CIS_NOALLOC_MAX_TOKENS (the array's every byte in use) at a small V,
    fp32 dlogits, some tokens masked; then a short call that reuses the array."""
    T, V = MAX_TOKENS, 64
    gen = torch.Generator().manual_seed(77)
    logits = (torch.randn((T, V), generator=gen) * 2.0).to(torch.bfloat16)
    ids = torch.randint(0, V, (T,), generator=gen, dtype=torch.int32)
    lp = torch.log_softmax(logits.float() + 0.3 * torch.randn((T, V), generator=gen),
                           dim=1).gather(1, ids.long()[:, None])[:, 0]
    adv = torch.where(torch.rand(T, generator=gen) < 0.5, -1.0, 1.0)
    mask = (torch.rand(T, generator=gen) > 0.1).to(torch.uint8)
    g = {k: v.cuda() for k, v in dict(logits=logits, ids=ids, lp=lp, adv=adv,
                                       mask=mask).items()}
    P = binding.cis_default_params("cis")
    ref = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                   dlogits_dtype=torch.float32)
    rc, out = _call(noalloc, g, P, T, V, dt=torch.float32)
    assert rc == binding.CIS_OK
    torch.cuda.synchronize()
    st = binding.decode_stats(out["stats"])
    assert st["status"] == 0 and st["n_valid"] == int(mask.sum()) and st["n_truncated"] > 0
    _same(out, ref)
    small = {k: v[:300] for k, v in g.items()}
    ref2 = binding.cis_loss_fwd_bwd(small["logits"], small["ids"], small["lp"], small["adv"], P,
                                    mask=small["mask"], dlogits_dtype=torch.float32)
    rc, out2 = _call(noalloc, small, P, 300, V, dt=torch.float32)
    assert rc == binding.CIS_OK
    torch.cuda.synchronize()
    _same(out2, ref2)


def test_noalloc_rejects_more_tokens_than_its_scratch(noalloc):
    P = binding.cis_default_params()
    fake = ctypes.c_void_p(0x10000)
    rc = noalloc(fake, binding.CIS_BF16, MAX_TOKENS + 1, 8, 8, fake, fake, None, fake, None,
                 None, 0, ctypes.byref(P), ctypes.c_void_p(0x4000000), binding.CIS_BF16, 8,
                 None, None, None, None, None, None, None)
    assert rc == binding.CIS_ERR_UNSUPPORTED


def test_noalloc_sequence_operator(noalloc):
    """Seq-MIS through the no-allocation entry point (forward pass, response
    weights, then the pass, all in the static array) equals the workspace
    entry point bit for bit."""
    b = synth.make_batch(1)
    g = _dev(b)
    P = binding.cis_default_params("seq_mis", lam=b.lam)
    B = b.cu_seqlens.shape[0] - 1
    rc, out = _call(noalloc, g, P, b.T, b.V, dt=torch.float32, cu=g["cu"], B=B)
    assert rc == 0
    ref = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                   cu_seqlens=g["cu"], dlogits_dtype=torch.float32)
    torch.cuda.synchronize()
    _same(out, ref)
