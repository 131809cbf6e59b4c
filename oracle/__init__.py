"""fp64 CPU oracle of the CIS token pass (arxiv 2609.32444).

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  The product
library never imports it and shares no code with it.

The arithmetic lives in ``cis_oracle.c`` (plain fp64 C, one row per host
thread).  This module compiles it on first use with the host C compiler and
marshals numpy arrays in and out.  Each function states the passage of the
paper it follows.

Pinned against the paper and mathematics (not against itself) by
``tests/test_oracle_pins.py``: tiny-V brute force at 50 digits, shift
invariance, normalisation, Lemma 3.1 (k = p + (1-p) e^eps from full inference
logits), Lemma B.2, Corollary B.6, Eq. 5, the special cases lambda = 0 and
lambda -> inf, the numbers the paper prints for lambda = 2.3, and central
finite differences of the loss against its gradient.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cis_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

MODE_CIS, MODE_TIS, MODE_EXACT, MODE_NONE = 0, 1, 2, 3
MODE_BAND, MODE_ICEPOP, MODE_KPOP, MODE_SEQ_TIS, MODE_SEQ_MIS = 4, 5, 6, 7, 8
SEQ_MODES = (MODE_SEQ_TIS, MODE_SEQ_MIS)
AGG_TOKEN_MEAN, AGG_SEQ_MEAN = 0, 1
F32, BF16 = 0, 1


class OracleParams(ctypes.Structure):
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
        ("n_global", ctypes.c_int64),
        ("g_global", ctypes.c_int64),
    ]


def params(mode=MODE_CIS, lam=2.3, kappa=5e-3, tis_cap=2.0, exact_lo=1e-6, exact_hi=1e6,
           clip_low=0.2, clip_high=0.28, agg=AGG_TOKEN_MEAN, icepop_lo=0.5, icepop_hi=5.0,
           kpop_phi=2.0, seq_cap=2.0, seq_lo=0.5, seq_hi=2.0, n_global=0,
           g_global=0) -> OracleParams:
    """Hyper-parameters; defaults are the deployed values of App. C.1 / Table 8.
    n_global / g_global (> 0): the batch's valid tokens / responses with a
    valid token when the rows passed are one shard of that batch."""
    return OracleParams(mode, agg, lam, kappa, tis_cap, exact_lo, exact_hi, clip_low, clip_high,
                        icepop_lo, icepop_hi, kpop_phi, seq_cap, seq_lo, seq_hi, n_global,
                        g_global)


def build(force: bool = False) -> str:
    """Compile cis_oracle.c into liboracle.so (host C compiler, OpenMP)."""
    with _lock:
        if (not force and os.path.exists(_LIB_PATH)
                and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
            return _LIB_PATH
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        P = ctypes.c_void_p
        i64, i32, dbl = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        lib.oracle_token_logprobs.argtypes = [P, i32, i64, i64, i64, P, P, P, P, ctypes.c_int]
        lib.oracle_token_logprobs.restype = ctypes.c_int
        lib.oracle_weights.argtypes = [P, P, P, i64, P, i64, ctypes.POINTER(OracleParams), P, P,
                                       P, P]
        lib.oracle_weights.restype = ctypes.c_int
        lib.oracle_loss_scales.argtypes = [P, i64, P, i64, ctypes.c_int, P]
        lib.oracle_loss_scales.restype = None
        lib.oracle_loss_fwd_bwd.argtypes = [
            P, i32, i64, i64, i64, P, P, P, P, P, P, i64, ctypes.POINTER(OracleParams), P,
            P, i64, P, P, P, P, P, P, P, P, P, P, ctypes.c_int]
        lib.oracle_loss_fwd_bwd.restype = ctypes.c_int
        lib.oracle_token_entropy.argtypes = [P, i32, i64, i64, i64, P, P, ctypes.c_int]
        lib.oracle_token_entropy.restype = None
        lib.oracle_mismatch_diagnostics.argtypes = [P, P, i32, i64, i64, i64, P, P,
                                                    ctypes.POINTER(OracleParams), P, P, P, P, P,
                                                    ctypes.c_int]
        lib.oracle_mismatch_diagnostics.restype = ctypes.c_int
        lib.oracle_binned_sums.argtypes = [P, P, i64, P, ctypes.c_int, P, ctypes.c_int, P, P]
        lib.oracle_binned_sums.restype = None
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = ctypes.c_int
        _ = dbl
        _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


F64 = 2


def _logits_arg(logits):
    """float32 [T, ld] -> F32; uint16 bf16 bit patterns -> BF16; float64 -> F64."""
    a = np.ascontiguousarray(logits)
    if a.dtype == np.float32:
        return a, F32
    if a.dtype == np.uint16:
        return a, BF16
    if a.dtype == np.float64:
        return a, F64
    raise TypeError(f"oracle logits must be float32, float64 or uint16 (bf16 bits), got {a.dtype}")


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact upcast of bf16 bit patterns (uint16) to float64."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _opt(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def token_logprobs(logits, ids, V=None, mask=None, nthreads=0):
    """log p_t = z_{t,y_t} - logsumexp(z_t) in fp64 (Sec. 2.1).  Returns (lp, lse, rc)."""
    lib = _load()
    a, dt = _logits_arg(logits)
    T, ld = a.shape
    V = ld if V is None else V
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    mask = _opt(mask, np.uint8)
    lp = np.zeros(T, np.float64)
    lse = np.zeros(T, np.float64)
    rc = lib.oracle_token_logprobs(_ptr(a), dt, T, V, ld, _ptr(ids), _ptr(mask), _ptr(lp),
                                   _ptr(lse), nthreads)
    return lp, lse, rc


def token_entropy(logits, V=None, mask=None, nthreads=0):
    """H_t = -sum_j p_tj log p_tj of each row's softmax in fp64 (App. D)."""
    lib = _load()
    a, dt = _logits_arg(logits)
    T, ld = a.shape
    V = ld if V is None else V
    mask = _opt(mask, np.uint8)
    h = np.zeros(T, np.float64)
    lib.oracle_token_entropy(_ptr(a), dt, T, V, ld, _ptr(mask), _ptr(h), nthreads)
    return h


def mismatch_diagnostics(z_train, z_infer, ids, P: OracleParams, mask=None, nthreads=0):
    """Per-position mismatch diagnostics in fp64 (App. A.5, Sec. 4.3 Fig. 5c-d):
    eps (Lemma 3.1's definition, normalised gauge), log k and p of the sampled
    token, and over y ~ q the squared bias ||E[(f - k) grad log p]||^2 and the
    variance increase of f grad log p over grad log p.  O(V^2) per position:
    small V only.  Returns a dict of [T] arrays."""
    lib = _load()
    a, dt = _logits_arg(z_train)
    b, dt2 = _logits_arg(z_infer)
    if dt != dt2 or a.shape != b.shape:
        raise ValueError("both logit tensors must have the same type and shape")
    T, V = a.shape
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    mask = _opt(mask, np.uint8)
    out = {k: np.zeros(T, np.float64) for k in ("eps", "logk", "p", "bias2", "dvar")}
    rc = lib.oracle_mismatch_diagnostics(_ptr(a), _ptr(b), dt, T, V, V, _ptr(ids), _ptr(mask),
                                         ctypes.byref(P), _ptr(out["eps"]), _ptr(out["logk"]),
                                         _ptr(out["p"]), _ptr(out["bias2"]), _ptr(out["dvar"]),
                                         nthreads)
    if rc != 0:
        raise ValueError("the diagnostics take a token operator")
    return out


def binned_sums(key, edges, values=(), mask=None):
    """Confidence-binned counts and fp64 sums (Sec. 4.3, Fig. 5b; App. A.5):
    token t (mask 1) in bin b when edges[b] <= key[t] < edges[b + 1], the last
    bin closed on the right; NaN or outside keys in no bin.  `key` and each
    value array are float32 of length T.  Returns (counts [nbins] int64,
    sums [len(values), nbins] float64)."""
    lib = _load()
    key = np.ascontiguousarray(key, dtype=np.float32)
    T = key.shape[0]
    edges = np.ascontiguousarray(edges, dtype=np.float64)
    nbins = edges.shape[0] - 1
    nv = len(values)
    vals = (np.ascontiguousarray(np.stack([np.asarray(v, np.float32) for v in values]))
            if nv else np.zeros((0, T), np.float32))
    mask = _opt(mask, np.uint8)
    counts = np.zeros(nbins, np.int64)
    sums = np.zeros((nv, nbins), np.float64)
    lib.oracle_binned_sums(_ptr(key), _ptr(mask), T, _ptr(edges), nbins, _ptr(vals), nv,
                           _ptr(counts), _ptr(sums))
    return counts, sums


def weights(lp_w, lp_inf, P: OracleParams, mask=None, cu_seqlens=None):
    """Algorithm 1 / Table 8 weights in fp64.  Returns (w, trunc, logk, eps).

    The sequence operators (Seq-TIS, Seq-MIS) need ``cu_seqlens`` (B + 1
    offsets of the responses)."""
    lib = _load()
    lp_w = np.ascontiguousarray(lp_w, dtype=np.float64)
    lp_inf = np.ascontiguousarray(lp_inf, dtype=np.float64)
    mask = _opt(mask, np.uint8)
    cu = _opt(cu_seqlens, np.int32)
    B = 0 if cu is None else cu.shape[0] - 1
    T = lp_w.shape[0]
    w = np.zeros(T, np.float64)
    tr = np.zeros(T, np.uint8)
    lk = np.zeros(T, np.float64)
    eps = np.zeros(T, np.float64)
    rc = lib.oracle_weights(_ptr(lp_w), _ptr(lp_inf), _ptr(mask), T, _ptr(cu), B,
                            ctypes.byref(P), _ptr(w), _ptr(tr), _ptr(lk), _ptr(eps))
    if rc != 0:
        raise ValueError("a sequence operator needs cu_seqlens")
    return w, tr, lk, eps


def loss_scales(T, mask=None, cu_seqlens=None, agg=AGG_TOKEN_MEAN):
    """Per-token normaliser s_t (Algorithm 1's 1/n, or Eq. 1's 1/(G |y_i|))."""
    lib = _load()
    mask = _opt(mask, np.uint8)
    cu = _opt(cu_seqlens, np.int32)
    B = 0 if cu is None else cu.shape[0] - 1
    s = np.zeros(T, np.float64)
    lib.oracle_loss_scales(_ptr(mask), T, _ptr(cu), B, agg, _ptr(s))
    return s


def loss_fwd_bwd(logits, ids, lp_inf, adv, P: OracleParams, V=None, lp_old=None, mask=None,
                 cu_seqlens=None, w_fixed=None, rows=None, want_dz=True, nthreads=0):
    """Weighted PPO-clipped token loss (Eq. 1, Algorithm 1) and d loss / d logits, fp64.

    ``rows``: indices of the rows whose dz is returned (None = all rows).
    Returns a dict with loss, terms, lp, lse, w, trunc, c, logk, dz
    ([len(rows), V] or [T, V]), stats and rc (0, or -1 when a valid row has an
    out-of-range id).  ``stats`` holds the batch statistics App. D logs and
    Lemma B.2's truncated excess: n_valid, n_truncated (valid tokens whose
    weight the operator changed), max_abs_logk (max over valid tokens of
    |log k|, tokens whose log k is not a number left out) and trunc_excess
    (sum over truncated tokens of k - w, k the token's own ratio).  The
    sequence operators need ``cu_seqlens``.
    """
    lib = _load()
    a, dt = _logits_arg(logits)
    T, ld = a.shape
    V = ld if V is None else V
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    lp_inf = np.ascontiguousarray(lp_inf, dtype=np.float64)
    adv = np.ascontiguousarray(adv, dtype=np.float64)
    lp_old = _opt(lp_old, np.float64)
    mask = _opt(mask, np.uint8)
    cu = _opt(cu_seqlens, np.int32)
    B = 0 if cu is None else cu.shape[0] - 1
    w_fixed = _opt(w_fixed, np.float64)
    rows_a = None if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    nrows = T if rows_a is None else rows_a.shape[0]
    dz = np.zeros((nrows, V), np.float64) if want_dz else None
    out = {k: np.zeros(T, np.float64) for k in ("lp", "lse", "w", "terms", "c", "logk")}
    trunc = np.zeros(T, np.uint8)
    loss = ctypes.c_double(0.0)
    stats = np.zeros(4, np.float64)
    rc = lib.oracle_loss_fwd_bwd(
        _ptr(a), dt, T, V, ld, _ptr(ids), _ptr(lp_inf), _ptr(lp_old), _ptr(adv), _ptr(mask),
        _ptr(cu), B, ctypes.byref(P), _ptr(w_fixed), _ptr(rows_a), nrows if rows_a is not None
        else 0, _ptr(dz), _ptr(out["lp"]), _ptr(out["lse"]), _ptr(out["w"]), _ptr(trunc),
        _ptr(out["terms"]), _ptr(out["c"]), ctypes.byref(loss), _ptr(out["logk"]), _ptr(stats),
        nthreads)
    if rc == -3:
        raise ValueError("a sequence operator needs cu_seqlens")
    out.update(loss=loss.value, trunc=trunc, dz=dz, rc=rc,
               stats=dict(n_valid=int(stats[0]), n_truncated=int(stats[1]),
                          max_abs_logk=float(stats[2]), trunc_excess=float(stats[3])))
    return out


def lmhead_fwd_bwd(hidden, weight, ids, lp_inf, adv, P: OracleParams, lp_old=None, mask=None,
                   rows=None, n_valid_total=None, w_fixed=None, want_dw=True, cu_seqlens=None):
    """The token pass through the LM head, in fp64.

    Logits z = H W^T (Sec. 2.1; the softmax is over these logits) are formed
    with an fp64 matrix product; the token pass itself is loss_fwd_bwd on those
    logits (Eq. 1, Algorithm 1, Table 8); the chain rule through z = H W^T gives
    dH = dz W and dW = dz^T H.

    ``hidden`` [T, H] and ``weight`` [V, H] as bf16 bit patterns (uint16) or
    float arrays.  ``rows``: evaluate only these tokens (their dH rows; dW then
    needs every valid token, so it is returned only when rows is None).  With a
    row subset and the token-mean normaliser, ``n_valid_total`` gives the number
    of valid tokens of the whole batch.
    """
    Hf = bf16_bits_to_f64(hidden) if np.asarray(hidden).dtype == np.uint16 else \
        np.asarray(hidden, np.float64)
    Wf = bf16_bits_to_f64(weight) if np.asarray(weight).dtype == np.uint16 else \
        np.asarray(weight, np.float64)
    if rows is not None and (P.mode in SEQ_MODES or cu_seqlens is not None):
        raise ValueError("row subsets cannot take whole responses")
    idx = np.arange(Hf.shape[0]) if rows is None else np.asarray(rows, np.int64)
    sel = lambda a: None if a is None else np.asarray(a)[idx]  # noqa: E731
    Z = Hf[idx] @ Wf.T
    out = loss_fwd_bwd(Z, sel(ids), sel(lp_inf), sel(adv), P, lp_old=sel(lp_old),
                       mask=sel(mask), w_fixed=sel(w_fixed), cu_seqlens=cu_seqlens)
    if rows is not None and n_valid_total is not None:
        if P.agg != AGG_TOKEN_MEAN:
            raise ValueError("row subsets need the token-mean normaliser")
        m = np.ones(len(idx), bool) if mask is None else np.asarray(mask)[idx].astype(bool)
        f = m.sum() / float(n_valid_total)
        for k in ("c", "terms", "dz"):
            out[k] = out[k] * f
        out["loss"] = float(out["terms"].sum())
    out["dhidden"] = out["dz"] @ Wf
    out["dhidden_abs"] = np.abs(out["dz"]) @ np.abs(Wf)
    if want_dw and rows is None:
        out["dweight"] = out["dz"].T @ Hf
        out["dweight_abs"] = np.abs(out["dz"]).T @ np.abs(Hf)
    out["logits"] = Z
    return out


def lmhead_token_groups(hidden, weight, ids, lp_inf, adv, P: OracleParams, lp_old=None,
                        mask=None, dh_rows=None, dw_rows=None, group=1024, nthreads=0):
    """The token pass through the LM head for batches whose logits do not fit
    in host memory at once (fp64 [T, V] is 20 GB at T=16384, V=151936).

    The same definitions as lmhead_fwd_bwd: z = H W^T in fp64 (Sec. 2.1), the
    token pass on those logits (Eq. 1, Algorithm 1, Table 8), and the chain
    rule through z = H W^T for the gradients.  Rows are independent, so the
    tokens are taken ``group`` at a time only to bound memory: each row's
    logits and results are those of the whole-batch computation; the token-mean
    normaliser uses the whole batch's count (n_global).

    Returns the per-token outputs of every token (lp, lse, w, trunc, c, terms,
    logk), the loss (their exact sum), the batch statistics, dH and |dz||W| on
    ``dh_rows`` (tokens) and dW and |dz|^T|H| on ``dw_rows`` (vocabulary
    rows): dW[v] = sum_t c_t (softmax_tv - [y_t = v]) H_t over every token.
    Token operators and the token-mean normaliser only (a group does not hold
    whole responses)."""
    import math
    if P.mode in SEQ_MODES or P.agg != AGG_TOKEN_MEAN:
        raise ValueError("token operators and the token-mean normaliser only")
    Hf = bf16_bits_to_f64(hidden) if np.asarray(hidden).dtype == np.uint16 else \
        np.asarray(hidden, np.float64)
    Wf = bf16_bits_to_f64(weight) if np.asarray(weight).dtype == np.uint16 else \
        np.asarray(weight, np.float64)
    T = Hf.shape[0]
    ids = np.asarray(ids, np.int32)
    m = np.ones(T, np.uint8) if mask is None else np.asarray(mask, np.uint8)
    n_valid = int(m.sum())
    Pg = OracleParams.from_buffer_copy(P)
    Pg.n_global = n_valid if P.n_global == 0 else P.n_global
    keys = ("lp", "lse", "w", "c", "terms", "logk")
    out = {k: np.zeros(T, np.float64) for k in keys}
    out["trunc"] = np.zeros(T, np.uint8)
    st = dict(n_valid=0, n_truncated=0, max_abs_logk=0.0, trunc_excess=0.0)
    rc = 0
    for g0 in range(0, T, group):
        g1 = min(T, g0 + group)
        Z = Hf[g0:g1] @ Wf.T
        r = loss_fwd_bwd(Z, ids[g0:g1], np.asarray(lp_inf)[g0:g1], np.asarray(adv)[g0:g1], Pg,
                         lp_old=None if lp_old is None else np.asarray(lp_old)[g0:g1],
                         mask=m[g0:g1], want_dz=False, nthreads=nthreads)
        del Z
        for k in keys + ("trunc",):
            out[k][g0:g1] = r[k]
        rs = r["stats"]
        st["n_valid"] += rs["n_valid"]
        st["n_truncated"] += rs["n_truncated"]
        st["max_abs_logk"] = max(st["max_abs_logk"], rs["max_abs_logk"])
        st["trunc_excess"] += rs["trunc_excess"]
        rc = rc or r["rc"]
    out["loss"] = math.fsum(out["terms"])
    out["stats"] = st
    out["rc"] = rc

    def dz_of(Zs, tok, cols):
        """dz[t, v] = c_t (exp(z_tv - lse_t) - [y_t = v]) for tokens tok, columns cols."""
        onehot = (ids[tok][:, None] == np.asarray(cols)[None, :]).astype(np.float64)
        c = out["c"][tok][:, None]
        live = (c != 0.0) & np.isfinite(out["lse"][tok])[:, None]  # masked rows: dz = 0
        with np.errstate(over="ignore", invalid="ignore"):
            d = c * (np.exp(Zs - out["lse"][tok][:, None]) - onehot)
        return np.where(live, d, 0.0)

    if dh_rows is not None:
        rows = np.asarray(dh_rows, np.int64)
        dz = dz_of(Hf[rows] @ Wf.T, rows, np.arange(Wf.shape[0]))
        out["dhidden"] = dz @ Wf
        out["dhidden_abs"] = np.abs(dz) @ np.abs(Wf)
    if dw_rows is not None:
        vs = np.asarray(dw_rows, np.int64)
        dz = dz_of(Hf @ Wf[vs].T, np.arange(T), vs)
        out["dweight"] = dz.T @ Hf
        out["dweight_abs"] = np.abs(dz).T @ np.abs(Hf)
    return out
