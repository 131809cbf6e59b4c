"""cis_loss_fwd_bwd_noalloc: the fused pass for callers that cannot allocate
device memory (framework extensions that get no allocator, C callers without
one).  It takes its scratch from a fixed array in the library's static device
memory instead of a caller workspace.

Checked through the C ABI against cis_loss_fwd_bwd on the same inputs, on two
calls in a row (the second call reuses the array the first one left behind),
within the tolerances the parity tests use.  This file is collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

from _util import bf16_tensor_bits, bf16_ulp_distance
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


def _call(f, g, P, T, V):
    dev = g["logits"].device
    out = {"dz": torch.full((T, V), float("nan"), dtype=torch.bfloat16, device=dev),
           "lp": torch.full((T,), float("nan"), device=dev),
           "w": torch.full((T,), float("nan"), device=dev),
           "trunc": torch.full((T,), 7, dtype=torch.uint8, device=dev),
           "stats": torch.zeros(ctypes.sizeof(binding.cis_stats_t), dtype=torch.uint8,
                                device=dev),
           "loss": torch.full((1,), float("nan"), dtype=torch.float64, device=dev)}
    ptr = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    rc = f(ptr(g["logits"]), binding.CIS_BF16, T, V, V, ptr(g["ids"]), ptr(g["lp"]), None,
           ptr(g["adv"]), ptr(g["mask"]), None, 0, ctypes.byref(P), ptr(out["dz"]),
           binding.CIS_BF16, V, ptr(out["lp"]), ptr(out["w"]), ptr(out["trunc"]), None,
           ptr(out["stats"]), ptr(out["loss"]),
           ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return rc, out


def test_noalloc_matches_workspace_entry_point_on_two_calls(noalloc):
    b = synth.make_batch(2, T=1024, V=32000)
    g = {k: v.cuda() for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv,
                                       mask=b.mask).items()}
    P = binding.cis_default_params("cis", lam=b.lam)
    ref = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"])
    torch.cuda.synchronize()
    # sum_t |loss term| = (1/n) sum_t w_t |A_t| here (no l_old, so rho = 1)
    ref_terms_scale = float((ref["w"] * g["adv"].abs()).sum().item()) / max(1, int(b.mask.sum()))
    for _ in range(2):
        rc, out = _call(noalloc, g, P, b.T, b.V)
        assert rc == binding.CIS_OK
        torch.cuda.synchronize()
        st = binding.decode_stats(out["stats"])
        assert st["status"] == 0
        lp_r, lp_o = ref["lp"].cpu().numpy(), out["lp"].cpu().numpy()
        assert np.all(np.abs(lp_o - lp_r) <= 2e-5 + 2.0 ** -21 * np.abs(lp_r))
        w_r, w_o = ref["w"].cpu().numpy(), out["w"].cpu().numpy()
        assert np.all(np.abs(w_o - w_r) <= 1e-5 * np.abs(w_r) + 1e-30)
        assert torch.equal(out["trunc"], ref["trunc"])
        d = bf16_ulp_distance(bf16_tensor_bits(out["dz"]), bf16_tensor_bits(ref["dlogits"]))
        assert d.max() <= 1
        lr, lo = float(ref["loss"].cpu()[0]), float(out["loss"].cpu()[0])
        assert abs(lo - lr) <= 1e-5 * ref_terms_scale + 1e-12
        assert st["n_valid"] == int(b.mask.sum())


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
    entry point."""
    b = synth.make_batch(1)
    g = {k: v.cuda() for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv,
                                       mask=b.mask, cu=b.cu_seqlens).items()}
    P = binding.cis_default_params("seq_mis", lam=b.lam)
    T, V = b.T, b.V
    dev = g["logits"].device
    dz = torch.empty((T, V), dtype=torch.float32, device=dev)
    w = torch.empty(T, device=dev)
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    ptr = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    rc = noalloc(ptr(g["logits"]), binding.CIS_F32, T, V, V, ptr(g["ids"]), ptr(g["lp"]), None,
                 ptr(g["adv"]), ptr(g["mask"]), ptr(g["cu"]), b.cu_seqlens.shape[0] - 1,
                 ctypes.byref(P), ptr(dz), binding.CIS_F32, V, None, ptr(w), None, None, None,
                 ptr(loss), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0
    ref = binding.cis_loss_fwd_bwd(g["logits"], g["ids"], g["lp"], g["adv"], P, mask=g["mask"],
                                   cu_seqlens=g["cu"], dlogits_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.equal(w, ref["w"]) and torch.equal(loss, ref["loss"])
    assert torch.equal(dz, ref["dlogits"])
