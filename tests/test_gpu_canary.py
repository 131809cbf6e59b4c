"""Guard bands around every output buffer of every entry point.

Each output (and each workspace) gets known bytes on both sides -- and, for a
dlogits matrix with a row stride wider than V, in the columns [V, ld_out) of
every row -- and after the call those bytes must be unchanged: no kernel may
write outside the memory its caller gave it.  Device buffers and, for the
host-buffer entry point, pinned host buffers.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_32444_gb300 import binding, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

GUARD = 4096  # bytes on each side
ALIGN = 1024  # start of each guarded interior


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


class Guarded:
    """`nbytes` of caller memory with GUARD bytes of a seeded pattern on each
    side (device memory, or pinned host memory when host=True)."""

    def __init__(self, nbytes, host=False, seed=0):
        self.n = int(nbytes)
        total = self.n + 2 * GUARD + ALIGN
        pat = np.random.default_rng(seed + self.n).integers(0, 256, total, dtype=np.uint8)
        buf = torch.from_numpy(pat)
        self.buf = buf.pin_memory() if host else buf.cuda()
        self.pattern = buf.clone()
        off = (-(self.buf.data_ptr() + GUARD)) % ALIGN
        self.lo, self.hi = off + GUARD, off + GUARD + self.n
        self.ptr = ctypes.c_void_p(self.buf.data_ptr() + self.lo)

    def view(self, dtype, shape):
        return self.buf[self.lo:self.hi].view(dtype).view(*shape)

    def check(self, name):
        torch.cuda.synchronize()
        got = self.buf.cpu()
        for a, b in ((0, self.lo), (self.hi, got.numel())):
            changed = int((got[a:b] != self.pattern[a:b]).sum())
            assert changed == 0, f"{name}: {changed} guard bytes written"


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _dev(t):
    return t.cuda().contiguous()


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _batch(V=4096, T=300):
    b = synth.make_batch(2, T=T, V=V)
    b.mask[::9] = 0
    return b


@pytest.mark.parametrize("pad,dz", [(8, torch.bfloat16), (3, torch.bfloat16), (4, torch.float32),
                                    (0, torch.float32)])
def test_fused_pass_writes_only_its_outputs(pad, dz):
    """cis_loss_fwd_bwd on the cluster path (16-byte rows) and the
    row-streaming path (a row stride of V + 3): dlogits rows and their padding
    columns, lp, w, trunc, entropy, stats, loss and the workspace."""
    b = _batch()
    T, V = b.T, b.V
    ld = V + pad
    es = torch.empty((), dtype=dz).element_size()
    L = binding.lib()
    dl = Guarded(T * ld * es, seed=1)
    outs = {k: Guarded(T * n, seed=2 + i) for i, (k, n) in
            enumerate((("lp", 4), ("w", 4), ("trunc", 1), ("ent", 4)))}
    stats = Guarded(ctypes.sizeof(binding.cis_stats_t), seed=7)
    loss = Guarded(8, seed=8)
    nws = binding.cis_loss_workspace_size(T, V)
    ws = Guarded(nws, seed=9)
    before = dl.buf.cpu().clone()
    P = binding.cis_default_params("cis", lam=b.lam)
    g = {k: _dev(v) for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv,
                                      mask=b.mask).items()}
    rc = L.cis_loss_fwd_bwd(_p(g["logits"]), binding.CIS_BF16, T, V, V, _p(g["ids"]), _p(g["lp"]),
                            None, _p(g["adv"]), _p(g["mask"]), None, 0, ctypes.byref(P), dl.ptr,
                            binding._dtype_code(dz), ld, outs["lp"].ptr, outs["w"].ptr,
                            outs["trunc"].ptr, outs["ent"].ptr, stats.ptr, loss.ptr, ws.ptr, nws,
                            _stream())
    assert rc == 0
    for nm, gb in dict(dlogits=dl, stats=stats, loss=loss, workspace=ws, **outs).items():
        gb.check(nm)
    after = dl.buf.cpu()[dl.lo:dl.hi].view(T, ld * es)
    assert torch.equal(after[:, V * es:], before[dl.lo:dl.hi].view(T, ld * es)[:, V * es:])
    assert binding.decode_stats(stats.view(torch.uint8, (stats.n,)))["status"] == 0


def test_forward_and_weights_write_only_their_outputs():
    b = _batch()
    T, V = b.T, b.V
    L = binding.lib()
    g = {k: _dev(v) for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer,
                                      mask=b.mask).items()}
    lp, lse, ent = (Guarded(4 * T, seed=s) for s in (11, 12, 13))
    rc = L.cis_token_logprobs(_p(g["logits"]), binding.CIS_BF16, T, V, V, _p(g["ids"]),
                              _p(g["mask"]), lp.ptr, lse.ptr, ent.ptr, None, _stream())
    assert rc == 0
    for nm, gb in dict(lp=lp, lse=lse, ent=ent).items():
        gb.check("token_logprobs " + nm)
    w, eps = Guarded(4 * T, seed=21), Guarded(4 * T, seed=22)
    tr = Guarded(T, seed=23)
    P = binding.cis_default_params("cis", lam=b.lam)
    rc = L.cis_weights(lp.ptr, _p(g["lp"]), _p(g["mask"]), T, None, 0, ctypes.byref(P), w.ptr,
                       tr.ptr, eps.ptr, _stream())
    assert rc == 0
    for nm, gb in dict(w=w, trunc=tr, eps=eps).items():
        gb.check("weights " + nm)
    cnt = Guarded(16, seed=24)
    cu = _dev(b.cu_seqlens)
    assert L.cis_count_valid(_p(g["mask"]), T, _p(cu), cu.numel() - 1, cnt.ptr, _stream()) == 0
    cnt.check("count_valid")


def test_host_path_writes_only_its_outputs():
    """cis_loss_fwd_bwd_host: pinned host outputs with guards, and its device
    workspace."""
    b = _batch(T=500)
    T, V = b.T, b.V
    L = binding.lib()
    dl = Guarded(T * V * 2, host=True, seed=31)
    outs = {k: Guarded(T * n, host=True, seed=32 + i) for i, (k, n) in
            enumerate((("lp", 4), ("w", 4), ("trunc", 1)))}
    stats = Guarded(ctypes.sizeof(binding.cis_stats_t), host=True, seed=36)
    loss = Guarded(8, host=True, seed=37)
    chunk = 128
    n = ctypes.c_size_t(0)
    assert L.cis_loss_host_workspace_size(T, V, binding.CIS_BF16, binding.CIS_BF16, chunk, 0,
                                          ctypes.byref(n)) == 0
    ws = Guarded(n.value, seed=38)
    h = {k: v.contiguous().pin_memory() for k, v in dict(logits=b.logits, ids=b.ids,
                                                          lp=b.lp_infer, adv=b.adv,
                                                          mask=b.mask).items()}
    P = binding.cis_default_params("cis", lam=b.lam)
    rc = L.cis_loss_fwd_bwd_host(_p(h["logits"]), binding.CIS_BF16, T, V, _p(h["ids"]),
                                 _p(h["lp"]), None, _p(h["adv"]), _p(h["mask"]), None, 0,
                                 ctypes.byref(P), dl.ptr, binding.CIS_BF16, outs["lp"].ptr,
                                 outs["w"].ptr, outs["trunc"].ptr, None, stats.ptr, loss.ptr,
                                 chunk, ws.ptr, n.value, _stream())
    assert rc == 0
    for nm, gb in dict(dlogits=dl, stats=stats, loss=loss, workspace=ws, **outs).items():
        gb.check("host " + nm)


@pytest.mark.parametrize("grad", [torch.float32, torch.bfloat16])
def test_lmhead_writes_only_its_outputs(grad):
    """cis_lmhead_fused with ragged token and vocabulary tiles (T=200, V=1000)
    and narrow vocabulary chunks: dH, dW, the per-token outputs and the
    workspace."""
    b = synth.make_batch(5, T=200, V=1000, H=256)
    T, V, H = 200, 1000, 256
    es = torch.empty((), dtype=grad).element_size()
    L = binding.lib()
    dh, dw = Guarded(T * H * es, seed=41), Guarded(V * H * es, seed=42)
    outs = {k: Guarded(T * n, seed=43 + i) for i, (k, n) in
            enumerate((("lp", 4), ("w", 4), ("trunc", 1), ("ent", 4)))}
    stats = Guarded(ctypes.sizeof(binding.cis_stats_t), seed=47)
    loss = Guarded(8, seed=48)
    nws = binding.cis_lmhead_workspace_size_chunk(T, V, H, 256)
    ws = Guarded(nws, seed=49)
    g = {k: _dev(v) for k, v in dict(h=b.hidden, w=b.weight, ids=b.ids, lp=b.lp_infer,
                                      adv=b.adv, mask=b.mask).items()}
    P = binding.cis_default_params("cis", lam=b.lam)
    rc = L.cis_lmhead_fused(_p(g["h"]), _p(g["w"]), T, H, V, _p(g["ids"]), _p(g["lp"]), None,
                            _p(g["adv"]), _p(g["mask"]), None, 0, ctypes.byref(P), dh.ptr,
                            dw.ptr, binding._dtype_code(grad), outs["lp"].ptr, outs["w"].ptr,
                            outs["trunc"].ptr, outs["ent"].ptr, stats.ptr, loss.ptr, ws.ptr, nws,
                            _stream())
    assert rc == 0
    for nm, gb in dict(dhidden=dh, dweight=dw, stats=stats, loss=loss, workspace=ws,
                       **outs).items():
        gb.check("lmhead " + nm)


@pytest.mark.parametrize("V", [4096, 1001])
def test_diagnostics_write_only_their_outputs(V):
    """cis_mismatch_diagnostics on the streaming kernel (bf16, V % 8 = 0) and
    the general kernel (V = 1001)."""
    T = 64
    gen = torch.Generator().manual_seed(5)
    zt = (torch.randn((T, V), generator=gen) * 2).to(torch.bfloat16).cuda()
    zi = (zt.float() + 0.1 * torch.randn((T, V), generator=gen).cuda()).to(torch.bfloat16)
    ids = torch.randint(0, V, (T,), generator=gen, dtype=torch.int32).cuda()
    L = binding.lib()
    outs = {k: Guarded(4 * T, seed=50 + i) for i, k in
            enumerate(("eps", "logk", "p", "bias2", "dvar"))}
    status = Guarded(4, seed=56)
    status.buf[status.lo:status.hi] = 0  # the caller clears the status word
    P = binding.cis_default_params("cis")
    rc = L.cis_mismatch_diagnostics(_p(zt), _p(zi), binding.CIS_BF16, T, V, V, V, _p(ids), None,
                                    ctypes.byref(P), outs["eps"].ptr, outs["logk"].ptr,
                                    outs["p"].ptr, outs["bias2"].ptr, outs["dvar"].ptr,
                                    status.ptr, _stream())
    assert rc == 0
    for nm, gb in dict(status=status, **outs).items():
        gb.check("diagnostics " + nm)


@pytest.mark.parametrize("T,nbins,nv", [(1000, 18, 2), (300000, 64, 4), (0, 3, 1)])
def test_binned_sums_write_only_their_outputs(T, nbins, nv):
    """cis_binned_sums: counts, sums and the workspace (the CTAs' partials and
    the ticket), one chunk a CTA and several."""
    rng = np.random.default_rng(T + nbins)
    key = torch.from_numpy(rng.random(T).astype(np.float32)).cuda()
    vals = [torch.from_numpy(rng.standard_normal(T).astype(np.float32)).cuda() for _ in range(nv)]
    L = binding.lib()
    need = ctypes.c_size_t()
    assert L.cis_binned_sums_workspace_size(T, nbins, nv, ctypes.byref(need)) == 0
    ws = Guarded(need.value, seed=71)
    counts = Guarded(8 * nbins, seed=72)
    sums = Guarded(8 * nbins * nv, seed=73)
    edges = np.linspace(0.0, 1.0, nbins + 1)
    earr = (ctypes.c_double * (nbins + 1))(*edges)
    varr = (ctypes.c_void_p * nv)(*[v.data_ptr() for v in vals])
    rc = L.cis_binned_sums(_p(key) if T else None, None, T, earr, nbins, varr, nv, counts.ptr,
                           sums.ptr, ws.ptr, need.value, _stream())
    assert rc == 0
    for nm, gb in dict(counts=counts, sums=sums, workspace=ws).items():
        gb.check("binned sums " + nm)


def test_noalloc_writes_only_its_outputs():
    """cis_loss_fwd_bwd_noalloc (scratch in the library's static array)."""
    b = _batch()
    T, V = b.T, b.V
    L = binding.lib()
    f = L.cis_loss_fwd_bwd_noalloc
    Pt, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    f.argtypes = [Pt, i32, i64, i64, i64, Pt, Pt, Pt, Pt, Pt, Pt, i64,
                  ctypes.POINTER(binding.cis_params_t), Pt, i32, i64, Pt, Pt, Pt, Pt, Pt, Pt, Pt]
    f.restype = ctypes.c_int
    dl = Guarded(T * V * 2, seed=61)
    outs = {k: Guarded(T * n, seed=62 + i) for i, (k, n) in
            enumerate((("lp", 4), ("w", 4), ("trunc", 1)))}
    stats = Guarded(ctypes.sizeof(binding.cis_stats_t), seed=66)
    loss = Guarded(8, seed=67)
    g = {k: _dev(v) for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv,
                                      mask=b.mask).items()}
    P = binding.cis_default_params("cis", lam=b.lam)
    rc = f(_p(g["logits"]), binding.CIS_BF16, T, V, V, _p(g["ids"]), _p(g["lp"]), None,
           _p(g["adv"]), _p(g["mask"]), None, 0, ctypes.byref(P), dl.ptr, binding.CIS_BF16, V,
           outs["lp"].ptr, outs["w"].ptr, outs["trunc"].ptr, None, stats.ptr, loss.ptr,
           _stream())
    assert rc == 0
    for nm, gb in dict(dlogits=dl, stats=stats, loss=loss, **outs).items():
        gb.check("noalloc " + nm)
