"""GPU parity of the confidence-binned counts and sums (Sec. 4.3, Fig. 5b;
App. A.5) against the fp64 oracle.

Counts must agree bit for bit: both sides compare the float32 key, widened to
fp64, with the same fp64 edges.  The sums add the same float32 values in fp64
in different orders, so a bin of n tokens may differ by at most the recursive
summation bound (n - 1) 2^-53 sum |v| (written here with a factor 2 of slack).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32444_gb300 import binding

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


def _compare(key, edges, values, mask=None):
    kd = torch.from_numpy(key).to(DEV)
    vd = [torch.from_numpy(v).to(DEV) for v in values]
    md = None if mask is None else torch.from_numpy(mask).to(DEV)
    counts, sums = binding.cis_binned_sums(kd, edges, vd, mask=md)
    torch.cuda.synchronize()
    rc, rs = oracle.binned_sums(key, edges, values, mask=mask)
    assert np.array_equal(counts.cpu().numpy(), rc)
    s = sums.cpu().numpy()
    for i, v in enumerate(values):
        _, abs_sum = oracle.binned_sums(key, edges, [np.abs(v)], mask=mask)
        tol = 2.0 * np.maximum(rc - 1, 0) * 2.0 ** -53 * abs_sum[0]
        assert np.all(np.abs(s[i] - rs[i]) <= tol), i
    return counts, sums


@pytest.mark.parametrize("T", [0, 1, 255, 256, 257, 5000, 300000])
def test_binned_sums_match_the_oracle(T):
    """Ragged and empty batches, one to three chunks a CTA (300000 tokens over
    1024 CTAs of 256), keys on the edges, NaN and out-of-range keys, masked
    tokens, four value arrays."""
    rng = np.random.default_rng(T + 3)
    edges = np.array([0.0, 0.05, 0.2, 0.3, 0.5, 0.565, 0.9, 0.99, 1.0],
                     np.float32).astype(np.float64)
    key = rng.uniform(-0.05, 1.05, T).astype(np.float32)
    if T >= 64:
        key[:9] = edges          # on the edges: the upper bin, the last edge closed
        key[9:64:7] = np.nan
    mask = (rng.random(T) < 0.9).astype(np.uint8)
    values = [rng.standard_normal(T).astype(np.float32),
              rng.exponential(3.0, T).astype(np.float32),
              (rng.standard_normal(T) * 1e4).astype(np.float32),
              np.ones(T, np.float32)]
    counts, sums = _compare(key, edges, values, mask)
    # the all-ones value counts the tokens once more
    assert np.array_equal(sums[3].cpu().numpy(), counts.cpu().numpy().astype(np.float64))


@pytest.mark.parametrize("nbins,nvalues", [(1, 0), (18, 2), (64, 4)])
def test_binned_sums_bin_and_value_counts(nbins, nvalues):
    """App. A.5's 18 logarithmic bins of 1 - p from 1.5e-6 to 0.68, one bin
    and the most bins; no values (counts only) up to four."""
    rng = np.random.default_rng(nbins)
    T = 20000
    one_minus_p = np.exp(rng.uniform(np.log(1e-7), np.log(0.9), T)).astype(np.float32)
    edges = np.geomspace(1.5e-6, 0.68, nbins + 1)
    values = [rng.standard_normal(T).astype(np.float32) for _ in range(nvalues)]
    _compare(one_minus_p, edges, values)


def test_binned_sums_are_deterministic():
    """Fixed-order sums: two calls give the same bits."""
    rng = np.random.default_rng(5)
    T = 100000
    key = torch.from_numpy(rng.random(T).astype(np.float32)).to(DEV)
    v = [torch.from_numpy(rng.standard_normal(T).astype(np.float32)).to(DEV) for _ in range(2)]
    edges = np.linspace(0.0, 1.0, 33)
    a = binding.cis_binned_sums(key, edges, v)
    b = binding.cis_binned_sums(key, edges, v)
    torch.cuda.synchronize()
    assert torch.equal(a[0], b[0])
    assert torch.equal(a[1].view(torch.int64), b[1].view(torch.int64))


def test_fig5b_truncation_bias_by_confidence():
    """Fig. 5b's quantity: the sampled tokens binned by p with k - f summed per
    bin, for CIS and TIS (C = 2), from the oracle's per-token weights on
    confidences log-uniform in [1e-4, 0.9999] (workload 3's range) and a log
    ratio N(0, 0.5^2).  The GPU bins them like the oracle, and below p = 0.565
    the CIS cap is looser than C = 2, so CIS removes no more weight there than
    TIS (Sec. 4.3)."""
    rng = np.random.default_rng(9)
    T = 4096
    lp = rng.uniform(np.log(1e-4), np.log(0.9999), T)
    lp_inf = lp - rng.normal(0.0, 0.5, T)
    edges = np.array([0.0, 0.1, 0.3, 0.565, 0.9, 0.99, 1.0])
    p = np.exp(lp).astype(np.float32)
    out = {}
    for name, mode in (("cis", oracle.MODE_CIS), ("tis", oracle.MODE_TIS)):
        w, tr, lk, _ = oracle.weights(lp, lp_inf, oracle.params(mode=mode, lam=2.3, tis_cap=2.0))
        kmf = (np.exp(lk) - w).astype(np.float32)
        counts, sums = _compare(p, edges, [kmf])
        out[name] = sums.cpu().numpy()[0]
    low = edges[1:] <= 0.565
    assert np.all(out["cis"][low] <= out["tis"][low] + 1e-6)
    assert out["tis"][low].sum() > 0  # TIS truncates there
