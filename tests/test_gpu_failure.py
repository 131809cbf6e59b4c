"""Failure detection on the GPU without a fault: a wait that nothing
completes runs out after its poll limit, the kernel reports
CIS_ERR_DEVICE_TIMEOUT in the device status word and ends, and the context
stays usable for the next call (which still matches the oracle)."""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2609_32444_gb300 import binding, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


@pytest.mark.parametrize("cluster_scope", [False, True])
def test_wait_runs_out_and_the_context_survives(cluster_scope):
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    binding.cis_selftest_bounded_wait(2000, cluster_scope, st)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert int(st.item()) == binding.CIS_ERR_DEVICE_TIMEOUT
    assert elapsed < 5.0  # 2000 polls of at most ~1 us each, plus the launch
    # the next call on the same context works and is right
    b = synth.make_batch(1)
    P = binding.cis_default_params("cis", lam=b.lam)
    out = binding.cis_loss_fwd_bwd(b.logits.to(DEV), b.ids.to(DEV), b.lp_infer.to(DEV),
                                   b.adv.to(DEV), P, mask=b.mask.to(DEV),
                                   dlogits_dtype=torch.float32)
    torch.cuda.synchronize()
    assert binding.decode_stats(out["stats"])["status"] == 0
    ref = oracle.loss_fwd_bwd(b.logits.numpy(), b.ids.numpy(), b.lp_infer.numpy(),
                              b.adv.numpy(), oracle.params(lam=b.lam), mask=b.mask.numpy())
    lp = out["lp"].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(lp - ref["lp"]) <= 2e-5 + 2.0 ** -21 * np.abs(ref["lp"]))
