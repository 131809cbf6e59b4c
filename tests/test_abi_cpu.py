"""Host-side tests of the C ABI: the library builds, loads, exports exactly the
functions include/*.h declares, and rejects bad arguments before touching the
GPU.  No compute call is made, so these run without a GPU."""
import ctypes
import glob
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and
                                not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="needs nvcc to build libcis")


@pytest.fixture(scope="module")
def binding():
    from paper_2609_32444_gb300 import build, binding as b
    build.build()
    b.lib()
    return b


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        names |= set(re.findall(r"CIS_API\s+[\w\s\*]+?\b(cis_\w+)\s*\(", src))
    return names


def test_exports_match_header(binding):
    declared = _declared()
    assert {"cis_loss_fwd_bwd", "cis_weights", "cis_token_logprobs"} <= declared
    out = subprocess.run(["nm", "-D", "--defined-only", binding.library_path()],
                         capture_output=True, text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if " T " in ln}
    exported = {n for n in exported if n.startswith("cis_")}
    assert exported == declared
    lib = binding.lib()
    for n in declared:
        assert hasattr(lib, n)


def test_default_params_are_the_papers(binding):
    p = binding.cis_default_params()
    assert (p.mode, p.agg) == (0, 0)
    assert (p.lam, p.kappa, p.tis_cap) == (2.3, 5e-3, 2.0)
    assert (p.exact_lo, p.exact_hi, p.clip_low, p.clip_high) == (1e-6, 1e6, 0.2, 0.28)


def test_status_strings(binding):
    for code in (0, 1, 2, 3, 4, 8):
        assert binding.status_string(code).startswith("CIS_")
    assert binding.status_string(12345) == "unknown cis status"


def test_workspace_size_grows_with_tokens(binding):
    a = binding.cis_loss_workspace_size(0, 10)
    b = binding.cis_loss_workspace_size(1000, 10)
    assert a >= 4 and b >= a + 1000 * (4 + 8 + 4 + 4 + 1)
    assert binding.lib().cis_loss_workspace_size(-1, 10, ctypes.byref(ctypes.c_size_t())) == 1


def _fwd_bwd_rc(binding, **over):
    """Call cis_loss_fwd_bwd with fake non-null pointers; validation must fail
    before any pointer is dereferenced or any kernel launched."""
    L = binding.lib()
    fake = ctypes.c_void_p(0x10000)
    ws = ctypes.c_void_p(0x20000)
    p = binding.cis_default_params()
    for k, v in over.pop("params", {}).items():
        setattr(p, k, v)
    args = dict(logits=fake, dtype=1, T=4, V=8, ld=8, ids=fake, lp_inf=fake, lp_old=None,
                adv=fake, mask=None, cu=None, B=0, dz=ctypes.c_void_p(0x40000), dz_dt=1,
                ld_out=8, ws=ws, ws_bytes=1 << 20)
    args.update(over)
    return L.cis_loss_fwd_bwd(args["logits"], args["dtype"], args["T"], args["V"], args["ld"],
                              args["ids"], args["lp_inf"], args["lp_old"], args["adv"],
                              args["mask"], args["cu"], args["B"], ctypes.byref(p), args["dz"],
                              args["dz_dt"], args["ld_out"], None, None, None, None, None, None,
                              args["ws"], args["ws_bytes"], None)


def test_lmhead_workspace_grows_with_the_chunk(binding):
    """2 ceil(T/128)*128 bytes per chunk column (dz in bf16); chunks wider
    than V (rounded up to 256) cost no more; a chunk must be a positive
    multiple of 256."""
    T, V, H = 1000, 5000, 512
    s256 = binding.cis_lmhead_workspace_size_chunk(T, V, H, 256)
    s512 = binding.cis_lmhead_workspace_size_chunk(T, V, H, 512)
    assert s512 - s256 in range(2 * 1024 * 256, 2 * 1024 * 256 + 1025)
    full = binding.cis_lmhead_workspace_size_chunk(T, V, H, 5120)
    assert binding.cis_lmhead_workspace_size_chunk(T, V, H, 1 << 20) == full
    assert binding.cis_lmhead_workspace_size(T, V, H) <= full
    for bad in (0, -256, 100, 384):
        with pytest.raises(RuntimeError):
            binding.cis_lmhead_workspace_size_chunk(T, V, H, bad)


@pytest.mark.parametrize("over", [
    dict(T=-1), dict(V=0), dict(ld=7), dict(ld_out=7), dict(dtype=5), dict(dz_dt=2),
    dict(logits=None), dict(ids=None), dict(lp_inf=None), dict(adv=None), dict(dz=None),
    dict(ws=None), dict(ws=ctypes.c_void_p(0x20010)), dict(ws_bytes=16),
    dict(params=dict(lam=-1.0)), dict(params=dict(kappa=1.5)), dict(params=dict(tis_cap=0.5)),
    dict(params=dict(exact_lo=0.0)), dict(params=dict(clip_low=1.0)),
    dict(params=dict(mode=9)), dict(params=dict(agg=1)),  # seq mean without cu_seqlens
    dict(params=dict(lam=float("nan"))),
    dict(dz=ctypes.c_void_p(0x10000 + 16)),  # dlogits overlaps the logits
])
def test_fwd_bwd_rejects_bad_arguments(binding, over):
    assert _fwd_bwd_rc(binding, **over) == 1


def test_other_entry_points_reject_bad_arguments(binding):
    L = binding.lib()
    fake = ctypes.c_void_p(0x10000)
    p = binding.cis_default_params()
    assert L.cis_token_logprobs(fake, 1, 4, 8, 7, fake, None, fake, None, None, None,
                                None) == 1
    assert L.cis_token_logprobs(None, 1, 4, 8, 8, fake, None, fake, None, None, None,
                                None) == 1
    assert L.cis_token_logprobs(fake, 1, 0, 8, 8, None, None, None, None, None, None,
                                None) == 0
    p.kappa = 2.0
    assert L.cis_weights(fake, fake, None, 4, None, 0, ctypes.byref(p), fake, None, None,
                         None) == 1
    p.kappa = 5e-3
    assert L.cis_weights(None, fake, None, 4, None, 0, ctypes.byref(p), fake, None, None,
                         None) == 1
    assert L.cis_weights(None, None, None, 0, None, 0, ctypes.byref(p), None, None, None,
                         None) == 0
    assert L.cis_default_params(None) == 1


@pytest.mark.parametrize("field,value", [("icepop_lo", 6.0), ("icepop_lo", -1.0),
                                         ("kpop_phi", -0.5), ("seq_cap", 0.0),
                                         ("seq_hi", 0.1), ("mode", 9)])
def test_new_operator_parameters_are_validated(binding, field, value):
    """Bands with lo > hi or lo < 0, a negative KPop threshold, a zero Seq-TIS
    cap and an unknown mode are refused before any GPU work."""
    L = binding.lib()
    fake = ctypes.c_void_p(0x10000)
    p = binding.cis_default_params("icepop")
    setattr(p, field, value)
    assert L.cis_weights(fake, fake, None, 4, None, 0, ctypes.byref(p), fake, None, None,
                         None) == 1


def test_sequence_operators_need_responses(binding):
    """Seq-TIS / Seq-MIS without cu_seqlens: CIS_ERR_INVALID_ARG before any
    GPU work, from the weights, the fused pass, the host path and the LM head."""
    L = binding.lib()
    fake = ctypes.c_void_p(0x10000)
    for mode in ("seq_tis", "seq_mis"):
        p = binding.cis_default_params(mode)
        assert L.cis_weights(fake, fake, None, 4, None, 0, ctypes.byref(p), fake, None, None,
                             None) == 1
        assert _fwd_bwd_rc(binding, params={"mode": binding.MODES[mode]}) == 1
    d = binding.cis_default_params()
    assert (d.icepop_lo, d.icepop_hi, d.kpop_phi) == (0.5, 5.0, 2.0)
    assert (d.seq_cap, d.seq_lo, d.seq_hi) == (2.0, 0.5, 2.0)


def test_binding_refuses_cpu_tensors(binding):
    import torch
    x = torch.zeros(2, 8)
    with pytest.raises(ValueError):
        binding.cis_token_logprobs(x, torch.zeros(2, dtype=torch.int32))


def test_selftest_bounded_wait_rejects_bad_arguments(binding):
    """The wait self-test validates on the host: a status word is required,
    the poll limit is 1 .. 2^21 and the scope 0 or 1 (no launch happens)."""
    L = binding.lib()
    dummy = ctypes.c_void_p(0x1000)  # never dereferenced: rejected first
    assert L.cis_selftest_bounded_wait(100, 0, None, None) == binding.CIS_ERR_INVALID_ARG
    assert L.cis_selftest_bounded_wait(0, 0, dummy, None) == binding.CIS_ERR_INVALID_ARG
    assert L.cis_selftest_bounded_wait((1 << 21) + 1, 0, dummy, None) == binding.CIS_ERR_INVALID_ARG
    assert L.cis_selftest_bounded_wait(100, 2, dummy, None) == binding.CIS_ERR_INVALID_ARG


def _bins_rc(binding, T=100, nbins=3, edges=(0.0, 0.25, 0.5, 1.0), nvalues=1, ws_bytes=1 << 20,
             ws=0x20000, key=0x10000, counts=0x30000, sums=0x40000, values=(0x50000,)):
    """cis_binned_sums with fake device pointers: every case here must fail
    host validation before the GPU is touched."""
    L = binding.lib()
    e = (ctypes.c_double * len(edges))(*edges)
    v = (ctypes.c_void_p * max(1, len(values)))(*values) if values is not None else None
    return L.cis_binned_sums(ctypes.c_void_p(key) if key else None, None, T, e, nbins, v,
                             nvalues, ctypes.c_void_p(counts) if counts else None,
                             ctypes.c_void_p(sums) if sums else None,
                             ctypes.c_void_p(ws) if ws else None, ws_bytes, None)


@pytest.mark.parametrize("over", [
    dict(T=-1), dict(nbins=0, edges=(0.0,)), dict(nbins=65, edges=tuple(range(66))),
    dict(nvalues=5, values=(0x50000,) * 5), dict(nvalues=-1),
    dict(edges=(0.0, 0.5, 0.5, 1.0)), dict(edges=(0.0, 0.7, 0.5, 1.0)),
    dict(edges=(0.0, float("nan"), 0.5, 1.0)), dict(key=0), dict(counts=0), dict(sums=0),
    dict(values=None), dict(ws=0), dict(ws=0x20010), dict(ws_bytes=64),
])
def test_binned_sums_host_validation(binding, over):
    assert _bins_rc(binding, **over) == 1  # CIS_ERR_INVALID_ARG


def test_binned_sums_workspace_size(binding):
    """256-byte blocks of fp64 partials for up to 1024 CTAs of 256 tokens, plus
    one block for the ticket."""
    L = binding.lib()
    n = ctypes.c_size_t()
    assert L.cis_binned_sums_workspace_size(0, 1, 0, ctypes.byref(n)) == 0
    assert n.value == 256 + 256
    assert L.cis_binned_sums_workspace_size(1 << 30, 64, 4, ctypes.byref(n)) == 0
    assert n.value == (1024 * 64 * 5 * 8 + 255) // 256 * 256 + 256
    for bad in ((-1, 1, 0), (10, 0, 0), (10, 65, 0), (10, 4, 5)):
        assert L.cis_binned_sums_workspace_size(*bad, ctypes.byref(n)) == 1
