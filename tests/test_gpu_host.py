"""cis_loss_fwd_bwd_host (host buffers, rows streamed through the GPU in
chunks) gives the outputs of cis_loss_fwd_bwd on the same batch."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_32444_gb300 import binding, synth

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_32444_gb300 import build
    build.build()
    binding.lib()


@pytest.mark.parametrize("cfg,T,V,chunk,agg", [(2, 1000, 32000, 256, 0), (2, 777, 4096, 100, 1),
                                              (1, 256, 1024, 96, 0), (3, 300, 151936, 64, 0)])
def test_host_path_equals_device_path(cfg, T, V, chunk, agg):
    b = synth.make_batch(cfg, T=T, V=V, device="cuda" if cfg == 3 else "cpu")
    P = binding.cis_default_params("cis", lam=b.lam, agg=agg)
    dz_dt = torch.bfloat16
    dev = {k: v.cuda() for k, v in dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv,
                                         mask=b.mask, cu=b.cu_seqlens).items()}
    ref = binding.cis_loss_fwd_bwd(dev["logits"], dev["ids"], dev["lp"], dev["adv"], P,
                                   mask=dev["mask"], cu_seqlens=dev["cu"] if agg else None,
                                   dlogits_dtype=dz_dt)
    host = {k: v.cpu().contiguous().pin_memory() for k, v in
            dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv, mask=b.mask,
                 cu=b.cu_seqlens).items()}
    dz_h = torch.empty((b.T, b.V), dtype=dz_dt).pin_memory()
    out = binding.cis_loss_fwd_bwd_host(host["logits"], host["ids"], host["lp"], host["adv"], P,
                                        dz_h, mask=host["mask"],
                                        cu_seqlens=host["cu"] if agg else None,
                                        chunk_tokens=chunk)
    torch.cuda.synchronize()
    assert torch.equal(dz_h.view(torch.int16), ref["dlogits"].cpu().view(torch.int16))
    assert torch.equal(out["lp"], ref["lp"].cpu())
    assert torch.equal(out["w"], ref["w"].cpu())
    assert torch.equal(out["trunc"], ref["trunc"].cpu())
    assert float(out["loss"][0]) == float(ref["loss"].cpu()[0])
    st = binding.decode_stats(out["stats"])
    assert st["status"] == 0 and st["n_valid"] == int(b.mask.sum())
    # the batch statistics are reduced once over the whole batch, as on the device
    assert st == binding.decode_stats(ref["stats"])
