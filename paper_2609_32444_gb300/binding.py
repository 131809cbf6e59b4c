"""Thin Python binding of libcis (include/cis.h), same names as the C ABI.

Argument marshalling only: tensors are passed as raw device pointers with the
current CUDA stream; every step of the token pass runs in libcis's kernels.
There is no CPU path -- importing works without a GPU, but every call needs
the compiled library and CUDA tensors, and raises otherwise.
"""

from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

CIS_OK, CIS_ERR_INVALID_ARG, CIS_ERR_UNSUPPORTED, CIS_ERR_CUDA = 0, 1, 2, 3
CIS_ERR_DEVICE_TIMEOUT, CIS_ERR_BAD_TOKEN_ID = 4, 8
CIS_F32, CIS_BF16 = 0, 1
CIS_MODE_CIS, CIS_MODE_TIS, CIS_MODE_EXACT, CIS_MODE_NONE = 0, 1, 2, 3
CIS_AGG_TOKEN_MEAN, CIS_AGG_SEQ_MEAN_TOKEN_MEAN = 0, 1

CIS_MODE_BAND, CIS_MODE_ICEPOP, CIS_MODE_KPOP, CIS_MODE_SEQ_TIS, CIS_MODE_SEQ_MIS = 4, 5, 6, 7, 8
MODES = {"cis": CIS_MODE_CIS, "tis": CIS_MODE_TIS, "exact": CIS_MODE_EXACT,
         "none": CIS_MODE_NONE, "band": CIS_MODE_BAND, "icepop": CIS_MODE_ICEPOP,
         "kpop": CIS_MODE_KPOP, "seq_tis": CIS_MODE_SEQ_TIS, "seq_mis": CIS_MODE_SEQ_MIS}
SEQ_MODES = ("seq_tis", "seq_mis")


class cis_params_t(ctypes.Structure):
    _fields_ = [
        ("mode", ctypes.c_int32),
        ("agg", ctypes.c_int32),
        ("lam", ctypes.c_double),
        ("kappa", ctypes.c_double),
        ("tis_cap", ctypes.c_double),
        ("exact_lo", ctypes.c_double),
        ("exact_hi", ctypes.c_double),
        ("clip_low", ctypes.c_double),
        ("clip_high", ctypes.c_double),
        ("icepop_lo", ctypes.c_double),
        ("icepop_hi", ctypes.c_double),
        ("kpop_phi", ctypes.c_double),
        ("seq_cap", ctypes.c_double),
        ("seq_lo", ctypes.c_double),
        ("seq_hi", ctypes.c_double),
        ("global_counts", ctypes.c_void_p),  # device int64 {N, G} of a sharded batch, or NULL
    ]


class cis_stats_t(ctypes.Structure):
    _fields_ = [
        ("loss", ctypes.c_double),
        ("trunc_excess", ctypes.c_double),
        ("n_valid", ctypes.c_int64),
        ("n_truncated", ctypes.c_int64),
        ("max_abs_logk", ctypes.c_float),
        ("status", ctypes.c_int32),
        ("entropy_sum", ctypes.c_double),
    ]


class CisError(RuntimeError):
    pass


_lib = None


def library_path() -> str:
    return _build.LIB_PATH


def lib():
    """The loaded libcis.so.  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB_PATH
    if not os.path.exists(path):
        raise ImportError(f"libcis.so is not built ({path}); run __graft_entry__.build()")
    L = ctypes.CDLL(path)
    P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    L.cis_default_params.argtypes = [ctypes.POINTER(cis_params_t)]
    L.cis_default_params.restype = ctypes.c_int
    L.cis_status_string.argtypes = [i32]
    L.cis_status_string.restype = ctypes.c_char_p
    L.cis_token_logprobs.argtypes = [P, i32, i64, i64, i64, P, P, P, P, P, P, P]
    L.cis_token_logprobs.restype = ctypes.c_int
    L.cis_weights.argtypes = [P, P, P, i64, P, i64, ctypes.POINTER(cis_params_t), P, P, P, P]
    L.cis_weights.restype = ctypes.c_int
    L.cis_loss_workspace_size.argtypes = [i64, i64, ctypes.POINTER(ctypes.c_size_t)]
    L.cis_loss_workspace_size.restype = ctypes.c_int
    L.cis_loss_fwd_bwd.argtypes = [P, i32, i64, i64, i64, P, P, P, P, P, P, i64,
                                   ctypes.POINTER(cis_params_t), P, i32, i64, P, P, P, P, P, P,
                                   P, ctypes.c_size_t, P]
    L.cis_loss_fwd_bwd.restype = ctypes.c_int
    L.cis_lmhead_workspace_size.argtypes = [i64, i64, i64, ctypes.POINTER(ctypes.c_size_t)]
    L.cis_lmhead_workspace_size.restype = ctypes.c_int
    L.cis_lmhead_workspace_size_chunk.argtypes = [i64, i64, i64, i64,
                                                  ctypes.POINTER(ctypes.c_size_t)]
    L.cis_lmhead_workspace_size_chunk.restype = ctypes.c_int
    L.cis_lmhead_fused.argtypes = [P, P, i64, i64, i64, P, P, P, P, P, P, i64,
                                   ctypes.POINTER(cis_params_t), P, P, i32, P, P, P, P, P, P,
                                   P, ctypes.c_size_t, P]
    L.cis_lmhead_fused.restype = ctypes.c_int
    L.cis_loss_host_workspace_size.argtypes = [i64, i64, i32, i32, i64, i64,
                                               ctypes.POINTER(ctypes.c_size_t)]
    L.cis_loss_host_workspace_size.restype = ctypes.c_int
    L.cis_loss_fwd_bwd_host.argtypes = [P, i32, i64, i64, P, P, P, P, P, P, i64,
                                        ctypes.POINTER(cis_params_t), P, i32, P, P, P, P, P, P,
                                        i64, P, ctypes.c_size_t, P]
    L.cis_loss_fwd_bwd_host.restype = ctypes.c_int
    L.cis_mismatch_diagnostics.argtypes = [P, P, i32, i64, i64, i64, i64, P, P,
                                           ctypes.POINTER(cis_params_t), P, P, P, P, P, P, P]
    L.cis_mismatch_diagnostics.restype = ctypes.c_int
    L.cis_count_valid.argtypes = [P, i64, P, i64, P, P]
    L.cis_count_valid.restype = ctypes.c_int
    L.cis_selftest_bounded_wait.argtypes = [ctypes.c_uint32, i32, P, P]
    L.cis_selftest_bounded_wait.restype = ctypes.c_int
    L.cis_profile_next_call.argtypes = [P, P]
    L.cis_profile_next_call.restype = ctypes.c_int
    L.cis_binned_sums_workspace_size.argtypes = [i64, i32, i32, ctypes.POINTER(ctypes.c_size_t)]
    L.cis_binned_sums_workspace_size.restype = ctypes.c_int
    L.cis_binned_sums.argtypes = [P, P, i64, ctypes.POINTER(ctypes.c_double), i32,
                                  ctypes.POINTER(ctypes.c_void_p), i32, P, P, P, ctypes.c_size_t,
                                  P]
    L.cis_binned_sums.restype = ctypes.c_int
    _lib = L
    return L


def status_string(code: int) -> str:
    return lib().cis_status_string(int(code)).decode()


def _check(rc: int, what: str):
    if rc != CIS_OK:
        raise CisError(f"{what}: {status_string(rc)}")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _dtype_code(dt) -> int:
    if dt == torch.bfloat16:
        return CIS_BF16
    if dt == torch.float32:
        return CIS_F32
    raise TypeError(f"unsupported dtype {dt}: libcis takes bfloat16 or float32")


def _need_cuda(*ts):
    for t in ts:
        if t is not None and not t.is_cuda:
            raise ValueError("libcis takes CUDA tensors")


def _rows(x: torch.Tensor):
    """(T, ld) of a 2-D tensor with unit column stride."""
    if x.dim() != 2 or (x.shape[1] > 1 and x.stride(1) != 1):
        raise ValueError("logits must be 2-D with contiguous rows")
    return x.shape[0], (x.stride(0) if x.shape[0] > 1 else x.shape[1])


def _vec(x, dtype, T, name):
    if x is None:
        return None
    if x.dtype != dtype or x.dim() != 1 or x.shape[0] != T or not x.is_contiguous():
        raise ValueError(f"{name} must be a contiguous [{T}] {dtype} tensor")
    return x


def cis_default_params(mode="cis", **kw) -> cis_params_t:
    """Defaults of App. C.1 / Table 8, with keyword overrides (lam, kappa, tis_cap,
    exact_lo, exact_hi, clip_low, clip_high, agg, icepop_lo, icepop_hi, kpop_phi,
    seq_cap, seq_lo, seq_hi)."""
    p = cis_params_t()
    _check(lib().cis_default_params(ctypes.byref(p)), "cis_default_params")
    p.mode = MODES[mode] if isinstance(mode, str) else int(mode)
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def cis_count_valid(T: int, mask=None, cu_seqlens=None, out=None) -> torch.Tensor:
    """This shard's {N, G} as a device int64 [2] tensor: valid tokens, and
    responses with a valid token (what a token-sharded run all-reduces)."""
    _need_cuda(mask, cu_seqlens)
    _vec(mask, torch.uint8, T, "mask")
    B = 0 if cu_seqlens is None else cu_seqlens.shape[0] - 1
    if out is None:
        dev = mask.device if mask is not None else (
            cu_seqlens.device if cu_seqlens is not None else torch.device("cuda"))
        out = torch.empty(2, dtype=torch.int64, device=dev)
    _need_cuda(out)
    _check(lib().cis_count_valid(_ptr(mask), T, _ptr(cu_seqlens), B, _ptr(out), _stream()),
           "cis_count_valid")
    return out


def with_global_counts(params: cis_params_t, counts: torch.Tensor) -> cis_params_t:
    """A copy of params whose normaliser uses the batch-wide {N, G} in
    `counts` (device int64 [2], kept alive by the caller until the call's
    kernels have run)."""
    _need_cuda(counts)
    if counts.dtype != torch.int64 or counts.numel() != 2 or not counts.is_contiguous():
        raise ValueError("counts must be a contiguous device int64 tensor of 2 elements")
    q = cis_params_t.from_buffer_copy(params)
    q.global_counts = counts.data_ptr()
    return q


def cis_token_logprobs(logits: torch.Tensor, ids: torch.Tensor, mask=None, V=None,
                       want_lse=False, dev_status=None, want_entropy=False):
    """log p of the sampled tokens (fp32) -- and the row logsumexp and the
    softmax entropy if asked: returns lp, or a tuple (lp, lse, entropy) with
    None for what was not asked when either is."""
    _need_cuda(logits, ids, mask)
    T, ld = _rows(logits)
    V = logits.shape[1] if V is None else V
    _vec(ids, torch.int32, T, "ids")
    _vec(mask, torch.uint8, T, "mask")
    lp = torch.empty(T, dtype=torch.float32, device=logits.device)
    lse = torch.empty(T, dtype=torch.float32, device=logits.device) if want_lse else None
    ent = torch.empty(T, dtype=torch.float32, device=logits.device) if want_entropy else None
    rc = lib().cis_token_logprobs(_ptr(logits), _dtype_code(logits.dtype), T, V, ld, _ptr(ids),
                                  _ptr(mask), _ptr(lp), _ptr(lse), _ptr(ent), _ptr(dev_status),
                                  _stream())
    _check(rc, "cis_token_logprobs")
    if want_entropy:
        return lp, lse, ent
    return (lp, lse) if want_lse else lp


def cis_weights(lp_train: torch.Tensor, lp_infer: torch.Tensor, params: cis_params_t,
                mask=None, want_trunc=True, want_eps=False, cu_seqlens=None):
    """Weights of Algorithm 1 / Table 8 (the sequence operators need
    cu_seqlens).  Returns (w, trunc or None, eps or None)."""
    _need_cuda(lp_train, lp_infer, mask, cu_seqlens)
    T = lp_train.shape[0]
    _vec(lp_train, torch.float32, T, "lp_train")
    _vec(lp_infer, torch.float32, T, "lp_infer")
    _vec(mask, torch.uint8, T, "mask")
    if cu_seqlens is not None and (cu_seqlens.dtype != torch.int32 or
                                   not cu_seqlens.is_contiguous()):
        raise TypeError("cu_seqlens must be contiguous int32")
    B = 0 if cu_seqlens is None else cu_seqlens.shape[0] - 1
    dev = lp_train.device
    w = torch.empty(T, dtype=torch.float32, device=dev)
    tr = torch.empty(T, dtype=torch.uint8, device=dev) if want_trunc else None
    eps = torch.empty(T, dtype=torch.float32, device=dev) if want_eps else None
    rc = lib().cis_weights(_ptr(lp_train), _ptr(lp_infer), _ptr(mask), T, _ptr(cu_seqlens), B,
                           ctypes.byref(params), _ptr(w), _ptr(tr), _ptr(eps), _stream())
    _check(rc, "cis_weights")
    return w, tr, eps


def cis_loss_workspace_size(T: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().cis_loss_workspace_size(T, V, ctypes.byref(n)), "cis_loss_workspace_size")
    return n.value


def cis_loss_fwd_bwd(logits: torch.Tensor, ids: torch.Tensor, lp_infer: torch.Tensor,
                     adv: torch.Tensor, params: cis_params_t, lp_old=None, mask=None,
                     cu_seqlens=None, dlogits=None, dlogits_dtype=None, V=None,
                     want_lp=True, want_w=True, want_trunc=True, workspace=None,
                     want_entropy=False):
    """Fused forward + backward token pass.  Returns a dict with dlogits, lp, w,
    trunc, entropy (if asked), loss (device fp64 [1]), stats (device bytes of
    cis_stats_t) and the workspace (its first int32 is the device status word)."""
    _need_cuda(logits, ids, lp_infer, adv, lp_old, mask, cu_seqlens, dlogits)
    T, ld = _rows(logits)
    V = logits.shape[1] if V is None else V
    dev = logits.device
    for x, dt, nm in ((ids, torch.int32, "ids"), (lp_infer, torch.float32, "lp_infer"),
                      (adv, torch.float32, "adv"), (lp_old, torch.float32, "lp_old"),
                      (mask, torch.uint8, "mask")):
        _vec(x, dt, T, nm)
    B = 0
    if cu_seqlens is not None:
        if cu_seqlens.dtype != torch.int32 or cu_seqlens.dim() != 1:
            raise ValueError("cu_seqlens must be int32 [B + 1]")
        B = cu_seqlens.shape[0] - 1
    if dlogits is None:
        dt = logits.dtype if dlogits_dtype is None else dlogits_dtype
        dlogits = torch.empty((T, V), dtype=dt, device=dev)
    To, ld_out = _rows(dlogits)
    if To != T or dlogits.shape[1] < V:
        raise ValueError("dlogits must be [T, >= V]")
    lp = torch.empty(T, dtype=torch.float32, device=dev) if want_lp else None
    w = torch.empty(T, dtype=torch.float32, device=dev) if want_w else None
    tr = torch.empty(T, dtype=torch.uint8, device=dev) if want_trunc else None
    ent = torch.empty(T, dtype=torch.float32, device=dev) if want_entropy else None
    stats = torch.empty(ctypes.sizeof(cis_stats_t), dtype=torch.uint8, device=dev)
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    nws = cis_loss_workspace_size(T, V)
    if workspace is None or workspace.numel() < nws:
        workspace = torch.empty(nws, dtype=torch.uint8, device=dev)
    rc = lib().cis_loss_fwd_bwd(
        _ptr(logits), _dtype_code(logits.dtype), T, V, ld, _ptr(ids), _ptr(lp_infer),
        _ptr(lp_old), _ptr(adv), _ptr(mask), _ptr(cu_seqlens), B, ctypes.byref(params),
        _ptr(dlogits), _dtype_code(dlogits.dtype), ld_out, _ptr(lp), _ptr(w), _ptr(tr),
        _ptr(ent), _ptr(stats), _ptr(loss), _ptr(workspace), workspace.numel(), _stream())
    _check(rc, "cis_loss_fwd_bwd")
    return {"dlogits": dlogits, "lp": lp, "w": w, "trunc": tr, "entropy": ent, "loss": loss,
            "stats": stats, "workspace": workspace}


def cis_loss_host_workspace_size(T, V, dtype, dlogits_dtype, chunk_tokens, B=0) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().cis_loss_host_workspace_size(T, V, _dtype_code(dtype), _dtype_code(dlogits_dtype),
                                              chunk_tokens, B, ctypes.byref(n)),
           "cis_loss_host_workspace_size")
    return n.value


def cis_loss_fwd_bwd_host(logits: torch.Tensor, ids: torch.Tensor, lp_infer: torch.Tensor,
                          adv: torch.Tensor, params: cis_params_t, dlogits: torch.Tensor,
                          lp_old=None, mask=None, cu_seqlens=None, chunk_tokens=512,
                          workspace=None, outputs=None, want_entropy=False):
    """The fused pass with every tensor in HOST memory (pinned for overlap);
    rows stream through the GPU in chunks.  ``outputs``: optional dict of host
    tensors lp, w, trunc, stats, loss to fill.  Returns that dict; it is valid
    after the current stream completes."""
    for x in (logits, ids, lp_infer, adv, dlogits, lp_old, mask, cu_seqlens):
        if x is not None and x.is_cuda:
            raise ValueError("cis_loss_fwd_bwd_host takes host tensors")
    if not (logits.is_contiguous() and dlogits.is_contiguous()):
        raise ValueError("logits and dlogits must be contiguous")
    T, V = logits.shape
    B = 0 if cu_seqlens is None else cu_seqlens.shape[0] - 1
    out = outputs or {}
    out.setdefault("lp", torch.empty(T, dtype=torch.float32).pin_memory())
    out.setdefault("w", torch.empty(T, dtype=torch.float32).pin_memory())
    out.setdefault("trunc", torch.empty(T, dtype=torch.uint8).pin_memory())
    if want_entropy:
        out.setdefault("entropy", torch.empty(T, dtype=torch.float32).pin_memory())
    out.setdefault("stats", torch.empty(ctypes.sizeof(cis_stats_t), dtype=torch.uint8).pin_memory())
    out.setdefault("loss", torch.empty(1, dtype=torch.float64).pin_memory())
    nws = cis_loss_host_workspace_size(T, V, logits.dtype, dlogits.dtype, chunk_tokens, B)
    if workspace is None or workspace.numel() < nws:
        workspace = torch.empty(nws, dtype=torch.uint8, device="cuda")
    rc = lib().cis_loss_fwd_bwd_host(
        _ptr(logits), _dtype_code(logits.dtype), T, V, _ptr(ids), _ptr(lp_infer), _ptr(lp_old),
        _ptr(adv), _ptr(mask), _ptr(cu_seqlens), B, ctypes.byref(params), _ptr(dlogits),
        _dtype_code(dlogits.dtype), _ptr(out["lp"]), _ptr(out["w"]), _ptr(out["trunc"]),
        _ptr(out.get("entropy")), _ptr(out["stats"]), _ptr(out["loss"]), chunk_tokens,
        _ptr(workspace), workspace.numel(),
        _stream())
    _check(rc, "cis_loss_fwd_bwd_host")
    out["workspace"] = workspace
    return out


def cis_lmhead_workspace_size(T: int, V: int, H: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().cis_lmhead_workspace_size(T, V, H, ctypes.byref(n)),
           "cis_lmhead_workspace_size")
    return n.value


def cis_lmhead_workspace_size_chunk(T: int, V: int, H: int, chunk: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().cis_lmhead_workspace_size_chunk(T, V, H, chunk, ctypes.byref(n)),
           "cis_lmhead_workspace_size_chunk")
    return n.value


def cis_lmhead_fused(hidden: torch.Tensor, weight: torch.Tensor, ids: torch.Tensor,
                     lp_infer: torch.Tensor, adv: torch.Tensor, params: cis_params_t,
                     lp_old=None, mask=None, cu_seqlens=None, grad_dtype=torch.float32,
                     workspace=None, chunk=None, want_entropy=False, dhidden=None,
                     dweight=None):
    """Token pass through the LM head (logits never stored).  `chunk` (a
    multiple of 256) sizes the workspace for vocabulary chunks of that many
    columns; by default the library's choice.  `dhidden` [T, H] and `dweight`
    [V, H] (contiguous, `grad_dtype`, 16-byte aligned) receive the gradients
    if given.  Returns a dict with dhidden, dweight, lp, w, trunc, loss, stats
    and the workspace."""
    _need_cuda(hidden, weight, ids, lp_infer, adv, lp_old, mask, cu_seqlens)
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise TypeError("hidden and weight must be bfloat16")
    if not (hidden.is_contiguous() and weight.is_contiguous()):
        raise ValueError("hidden and weight must be contiguous")
    T, H = hidden.shape
    V = weight.shape[0]
    if weight.shape[1] != H:
        raise ValueError("weight must be [V, H]")
    dev = hidden.device
    for x, dt, nm in ((ids, torch.int32, "ids"), (lp_infer, torch.float32, "lp_infer"),
                      (adv, torch.float32, "adv"), (lp_old, torch.float32, "lp_old"),
                      (mask, torch.uint8, "mask")):
        _vec(x, dt, T, nm)
    B = 0 if cu_seqlens is None else cu_seqlens.shape[0] - 1
    def _out(x, shape, nm):
        if x is None:
            return torch.empty(shape, dtype=grad_dtype, device=dev)
        if x.dtype != grad_dtype or tuple(x.shape) != shape or not x.is_contiguous():
            raise ValueError(f"{nm} must be a contiguous {grad_dtype} tensor of shape {shape}")
        _need_cuda(x)
        return x

    dh = _out(dhidden, (T, H), "dhidden")
    dw = _out(dweight, (V, H), "dweight")
    lp = torch.empty(T, dtype=torch.float32, device=dev)
    w = torch.empty(T, dtype=torch.float32, device=dev)
    tr = torch.empty(T, dtype=torch.uint8, device=dev)
    ent = torch.empty(T, dtype=torch.float32, device=dev) if want_entropy else None
    stats = torch.empty(ctypes.sizeof(cis_stats_t), dtype=torch.uint8, device=dev)
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    if workspace is None:  # else the caller's, as given (the library checks its size)
        need = (cis_lmhead_workspace_size(T, V, H) if chunk is None
                else cis_lmhead_workspace_size_chunk(T, V, H, chunk))
        workspace = torch.empty(need + 1024, dtype=torch.uint8, device=dev)
        off = (-workspace.data_ptr()) % 1024  # 1024-byte aligned start
        ws = workspace[off:off + need]
    else:
        ws = workspace
    rc = lib().cis_lmhead_fused(
        _ptr(hidden), _ptr(weight), T, H, V, _ptr(ids), _ptr(lp_infer), _ptr(lp_old),
        _ptr(adv), _ptr(mask), _ptr(cu_seqlens), B, ctypes.byref(params), _ptr(dh), _ptr(dw),
        _dtype_code(grad_dtype), _ptr(lp), _ptr(w), _ptr(tr), _ptr(ent), _ptr(stats),
        _ptr(loss), _ptr(ws), ws.numel(), _stream())
    _check(rc, "cis_lmhead_fused")
    return {"dhidden": dh, "dweight": dw, "lp": lp, "w": w, "trunc": tr, "entropy": ent,
            "loss": loss, "stats": stats, "workspace": ws}


def cis_mismatch_diagnostics(logits_train: torch.Tensor, logits_infer: torch.Tensor,
                             ids: torch.Tensor, params: cis_params_t, mask=None, V=None,
                             dev_status=None):
    """Per-position mismatch diagnostics (App. A.5; Sec. 4.3, Fig. 5c-d): a dict
    of device float [T] tensors eps, logk, p, bias2, dvar."""
    _need_cuda(logits_train, logits_infer, ids, mask)
    if logits_train.dtype != logits_infer.dtype:
        raise TypeError("both logit tensors must have the same type")
    T, ld_t = _rows(logits_train)
    Ti, ld_i = _rows(logits_infer)
    if Ti != T:
        raise ValueError("both logit tensors must have T rows")
    V = min(logits_train.shape[1], logits_infer.shape[1]) if V is None else V
    _vec(ids, torch.int32, T, "ids")
    _vec(mask, torch.uint8, T, "mask")
    out = {k: torch.empty(T, dtype=torch.float32, device=logits_train.device)
           for k in ("eps", "logk", "p", "bias2", "dvar")}
    rc = lib().cis_mismatch_diagnostics(
        _ptr(logits_train), _ptr(logits_infer), _dtype_code(logits_train.dtype), T, V, ld_t, ld_i,
        _ptr(ids), _ptr(mask), ctypes.byref(params), _ptr(out["eps"]), _ptr(out["logk"]),
        _ptr(out["p"]), _ptr(out["bias2"]), _ptr(out["dvar"]), _ptr(dev_status), _stream())
    _check(rc, "cis_mismatch_diagnostics")
    return out


def cis_binned_sums(key: torch.Tensor, edges, values=(), mask=None):
    """Confidence-binned counts and fp64 sums (Sec. 4.3, Fig. 5b; App. A.5):
    `key` and each of `values` are device float [T] tensors, `edges` a
    sequence of nbins + 1 strictly ascending floats.  Returns (counts int64
    [nbins], sums float64 [len(values), nbins]) on the device."""
    _need_cuda(key, mask, *values)
    T = key.shape[0]
    _vec(key, torch.float32, T, "key")
    _vec(mask, torch.uint8, T, "mask")
    for i, v in enumerate(values):
        _vec(v, torch.float32, T, f"values[{i}]")
    e = [float(x) for x in edges]
    nb, nv = len(e) - 1, len(values)
    need = ctypes.c_size_t(0)
    _check(lib().cis_binned_sums_workspace_size(T, nb, nv, ctypes.byref(need)),
           "cis_binned_sums_workspace_size")
    wbuf = torch.empty(need.value + 256, dtype=torch.uint8, device=key.device)
    ws = wbuf[(-wbuf.data_ptr()) % 256:][:need.value]
    counts = torch.empty(nb, dtype=torch.int64, device=key.device)
    sums = torch.empty((nv, nb), dtype=torch.float64, device=key.device)
    earr = (ctypes.c_double * len(e))(*e)
    varr = (ctypes.c_void_p * max(nv, 1))(*[v.data_ptr() for v in values])
    rc = lib().cis_binned_sums(_ptr(key), _ptr(mask), T, earr, nb, varr if nv else None, nv,
                               _ptr(counts), _ptr(sums) if nv else None, _ptr(ws), ws.numel(),
                               _stream())
    _check(rc, "cis_binned_sums")
    return counts, sums


def cis_selftest_bounded_wait(max_polls: int, cluster_scope: bool = False,
                              dev_status: "torch.Tensor | None" = None) -> torch.Tensor:
    """Run the bounded-wait self-test (a wait that nothing completes, with a
    limit of max_polls polls); returns the device status word (int32 [1]),
    which then carries CIS_ERR_DEVICE_TIMEOUT."""
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device="cuda")
    _need_cuda(dev_status)
    _check(lib().cis_selftest_bounded_wait(int(max_polls), int(bool(cluster_scope)),
                                           _ptr(dev_status), _stream()),
           "cis_selftest_bounded_wait")
    return dev_status


def cis_profile_next_call(begin: "torch.cuda.Event | None", end: "torch.cuda.Event | None"):
    """Have the next cis_loss_fwd_bwd on this thread record these events around
    its main kernel (timing aid; the call does the same work)."""
    b = None if begin is None else ctypes.c_void_p(begin.cuda_event)
    e = None if end is None else ctypes.c_void_p(end.cuda_event)
    if (begin is not None and not b.value) or (end is not None and not e.value):
        raise ValueError("record the events once first: torch creates them lazily")
    _check(lib().cis_profile_next_call(b, e), "cis_profile_next_call")


def decode_stats(stats: torch.Tensor) -> dict:
    """Read a cis_stats_t written on the device (synchronises)."""
    raw = bytes(stats.cpu().numpy().tobytes())
    s = cis_stats_t.from_buffer_copy(raw)
    return {f: getattr(s, f) for f, _ in cis_stats_t._fields_}


def device_status(workspace: torch.Tensor) -> int:
    """The device status word of the last call that used this workspace."""
    return int(workspace[:4].view(torch.int32).item())
