"""Seeded synthetic inputs for the CIS token pass.

The paper trains MoE policies on GSM8K rollouts (Sec. 4.1); neither the models
nor the rollouts exist here, so every workload is synthetic, with the value
distributions the paper reports for the mismatch (App. A: a narrow body of
per-logit perturbations with a heavy tail, 68-85% of tokens at p > 0.99,
responses of a few hundred tokens, binary rewards normalised within groups).

This module only draws inputs.  It holds none of the method's arithmetic: the
training-side log-softmax, the weight, the loss and the gradient are computed
by the library (and, independently, by the oracle).  Two things the method
takes as INPUTS are simulated here the way an inference engine produces them:
the sampled token (Gumbel-max over the inference logits) and the log-probability
the inference engine records for it (fp32 log-softmax of the inference logits).

Workloads (``cfg`` ids):
  1  T=256 (4 x 64), V=1024, fp32 logits ~ N(0, 2^2); inference logits = z +
     N(0, 0.05^2), 1% of tokens get +4 on one uniformly chosen logit; advantages
     +-1 per response; all valid; CIS threshold lambda = 1.0.
  2  T=4096, V=32000, bf16 logits ~ N(0, 3^2), 10% of rows get +12 on one
     logit; 32 responses, lengths U[32, 256] scaled down to fit, right padding
     masked; perturbation N(0, 0.1^2) per logit plus, on 0.5% of tokens, a
     Student-t(2) * 0.5 draw on every logit of the row; groups of 8, rewards
     Bernoulli(0.4).
  3  T=16384 (64 x 256), V=151936, bf16; per row a temperature is found by
     bisection so that the top probability equals p* ~ LogUniform[1e-4,
     0.9999]; perturbation N(0, 0.15^2); groups of 8, rewards Bernoulli(0.5).
  4  T=65536, V=151936, bf16; 32 responses, lengths U[512, 4096] rescaled so
     that exactly 40% of the slots are right padding (masked); rows as in 3,
     plus on 1% of valid tokens the inference logit of the sampled token is
     lowered by 6, which raises eps by exactly 6 (Lemma 3.1).
  5  hidden [16384, 2048] bf16 ~ N(0, 1), unembedding W [151936, 2048] bf16 ~
     N(0, 0.02^2); logits H W^T; inference side and advantages as in 3.

``T``/``V`` overrides keep a workload's recipe at a smaller size (the sizes the
oracle finishes in seconds).  Seeds default to 1000 + cfg.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

WORKLOADS = {
    1: dict(name="c1_t256_v1024_f32", T=256, V=1024, dtype="f32", lam=1.0),
    2: dict(name="c2_t4096_v32000_bf16", T=4096, V=32000, dtype="bf16", lam=2.3),
    3: dict(name="c3_t16384_v151936_bf16", T=16384, V=151936, dtype="bf16", lam=2.3),
    4: dict(name="c4_t65536_v151936_bf16_masked40", T=65536, V=151936, dtype="bf16", lam=2.3),
    5: dict(name="c5_lmhead_t16384_h2048_v151936_bf16", T=16384, V=151936, H=2048,
            dtype="bf16", lam=2.3),
    # the mismatch diagnostics: workload 3's recipe, keeping both engines' logits
    6: dict(name="c6_mismatch_t16384_v151936_bf16", T=16384, V=151936, dtype="bf16", lam=2.3),
}


@dataclass
class Batch:
    """One synthetic batch.  Tensors live on ``device``."""
    cfg: int
    T: int
    V: int
    logits: torch.Tensor | None       # [T, V] f32 or bf16 (None for cfg 5)
    ids: torch.Tensor                  # int32 [T]
    lp_infer: torch.Tensor             # f32 [T]
    adv: torch.Tensor                  # f32 [T]
    mask: torch.Tensor                 # uint8 [T]
    cu_seqlens: torch.Tensor           # int32 [B + 1]
    lam: float
    hidden: torch.Tensor | None = None  # cfg 5: [T, H] bf16
    weight: torch.Tensor | None = None  # cfg 5: [V, H] bf16
    extra: dict = field(default_factory=dict)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _gumbel_argmax(x: torch.Tensor, g: torch.Generator) -> torch.Tensor:
    """A sample of softmax(x) per row (Gumbel-max)."""
    u = torch.rand(x.shape, generator=g, device=x.device, dtype=torch.float32)
    u = u.clamp_(min=1e-20, max=1.0 - 1e-7)
    return torch.argmax(x - torch.log(-torch.log(u)), dim=1)


def _engine_logprob(x: torch.Tensor, ids: torch.Tensor) -> torch.Tensor:
    """What an inference engine records for the sampled token: fp32 log-softmax."""
    x = x.float()
    return (torch.gather(x, 1, ids.view(-1, 1)).view(-1) - torch.logsumexp(x, dim=1))


def _group_advantages(rewards: torch.Tensor, group: int) -> torch.Tensor:
    """(r - mean_g) / (std_g + 1e-6), population std, 0 for a constant group."""
    r = rewards.view(-1, group).double()
    mu = r.mean(dim=1, keepdim=True)
    sd = r.std(dim=1, unbiased=False, keepdim=True)
    a = torch.where(sd > 0, (r - mu) / (sd + 1e-6), torch.zeros_like(r))
    return a.view(-1).float()


def _pack(lengths: list[int], T: int, seq_adv: torch.Tensor, device):
    """Pack responses back to back from token 0; the rest is masked padding."""
    cu = [0]
    for n in lengths:
        cu.append(cu[-1] + n)
    assert cu[-1] <= T
    mask = torch.zeros(T, dtype=torch.uint8)
    adv = torch.zeros(T, dtype=torch.float32)
    for i, n in enumerate(lengths):
        mask[cu[i]:cu[i + 1]] = 1
        adv[cu[i]:cu[i + 1]] = float(seq_adv[i])
    return (torch.tensor(cu, dtype=torch.int32, device=device), mask.to(device),
            adv.to(device))


def _scale_lengths(raw: list[int], total: int) -> list[int]:
    """Scale lengths so they sum to exactly ``total`` (largest remainders)."""
    s = sum(raw)
    exact = [n * total / s for n in raw]
    out = [int(math.floor(e)) for e in exact]
    rem = total - sum(out)
    order = sorted(range(len(raw)), key=lambda i: exact[i] - out[i], reverse=True)
    for i in order[:rem]:
        out[i] += 1
    return out


def _tempered_rows(n: int, V: int, pstar: torch.Tensor, g: torch.Generator, device,
                   iters: int = 48) -> torch.Tensor:
    """Rows u/tau with u ~ N(0,1)^V and tau set by bisection so that the top
    probability of softmax(u/tau) equals p* (per row)."""
    u = torch.randn((n, V), generator=g, device=device, dtype=torch.float32)
    d = u - u.max(dim=1, keepdim=True).values            # <= 0, top entry 0
    target = -torch.log(pstar.double()).float()            # logsumexp(d/tau) = -log p*
    lo = torch.full((n,), math.log(1e-4), device=device)
    hi = torch.full((n,), math.log(1e3), device=device)
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        f = torch.logsumexp(d / torch.exp(mid).view(-1, 1), dim=1)
        too_hot = f > target                                # tau too large
        hi = torch.where(too_hot, mid, hi)
        lo = torch.where(too_hot, lo, mid)
    tau = torch.exp(0.5 * (lo + hi)).view(-1, 1)
    return u / tau


def make_batch(cfg: int, device="cpu", seed: int | None = None, T: int | None = None,
               V: int | None = None, chunk_rows: int = 1024, H: int | None = None,
               keep_infer: bool = False) -> Batch:
    """Draw the synthetic batch of workload ``cfg`` (see module docstring).
    ``keep_infer`` (workloads 1-4; always for 6) also returns the inference
    engine's logits, rounded to the batch's logit type, as
    ``extra["logits_infer"]``."""
    if cfg == 6:
        b = make_batch(3, device, 1006 if seed is None else seed, T, V, chunk_rows,
                       keep_infer=True)
        b.cfg = 6
        return b
    spec = WORKLOADS[cfg]
    T = spec["T"] if T is None else T
    V = spec["V"] if V is None else V
    seed = 1000 + cfg if seed is None else seed
    device = torch.device(device)
    g = _gen(seed, device)
    gcpu = _gen(seed + 7919, "cpu")          # small host-side draws (lengths, rewards)

    if cfg == 1:
        z = torch.randn((T, V), generator=g, device=device) * 2.0
        zi = z + torch.randn((T, V), generator=g, device=device) * 0.05
        n_out = max(1, round(0.01 * T))
        rows = torch.randperm(T, generator=gcpu)[:n_out].to(device)
        cols = torch.randint(0, V, (n_out,), generator=gcpu).to(device)
        zi[rows, cols] += 4.0
        ids = _gumbel_argmax(zi, g)
        lp_inf = _engine_logprob(zi, ids)
        nseq = 4
        L = T // nseq
        signs = torch.tensor([1.0, -1.0] * (nseq // 2))[torch.randperm(nseq, generator=gcpu)]
        cu, mask, adv = _pack([L] * nseq, T, signs, device)
        extra = {"logits_infer": zi.float().contiguous()} if keep_infer else {}
        return Batch(cfg, T, V, z.float().contiguous(), ids.int(), lp_inf, adv, mask, cu,
                     spec["lam"], extra=extra)

    if cfg == 2:
        z = torch.randn((T, V), generator=g, device=device) * 3.0
        n_dom = round(0.10 * T)
        rows = torch.randperm(T, generator=gcpu)[:n_dom].to(device)
        cols = torch.randint(0, V, (n_dom,), generator=gcpu).to(device)
        z[rows, cols] += 12.0
        z = z.to(torch.bfloat16)
        zi = z.float() + torch.randn((T, V), generator=g, device=device) * 0.1
        n_t = max(1, round(0.005 * T))
        trows = torch.randperm(T, generator=gcpu)[:n_t].to(device)
        # Student-t with 2 degrees of freedom: N / sqrt(chi2_2 / 2), chi2_2 / 2 ~ Exp(1)
        nrm = torch.randn((n_t, V), generator=g, device=device)
        ex = -torch.log(torch.rand((n_t, V), generator=g, device=device).clamp_(min=1e-30))
        tdraw = nrm / torch.sqrt(ex) * 0.5
        zi[trows] += tdraw
        ids = _gumbel_argmax(zi, g)
        lp_inf = _engine_logprob(zi, ids)
        nseq = 32
        raw = torch.randint(32, 257, (nseq,), generator=gcpu).tolist()
        lengths = raw if sum(raw) <= T else _scale_lengths(raw, T)
        rewards = (torch.rand(nseq, generator=gcpu) < 0.4).float()
        cu, mask, adv = _pack(lengths, T, _group_advantages(rewards, 8), device)
        extra = {"logits_infer": zi.to(torch.bfloat16).contiguous()} if keep_infer else {}
        return Batch(cfg, T, V, z.contiguous(), ids.int(), lp_inf, adv, mask, cu, spec["lam"],
                     extra=extra)

    if cfg in (3, 4, 5):
        if cfg == 4:
            nseq = 32
            raw = torch.randint(512, 4097, (nseq,), generator=gcpu).tolist()
            lengths = _scale_lengths(raw, int(round(0.6 * T)))
        else:
            nseq = max(8, (T // 256) // 8 * 8) if T >= 2048 else 8
            base, rem = divmod(T, nseq)
            lengths = [base + (1 if i < rem else 0) for i in range(nseq)]
        rewards = (torch.rand(nseq, generator=gcpu) < 0.5).float()
        cu, mask, adv = _pack(lengths, T, _group_advantages(rewards, 8), device)

        if cfg == 5:
            H = spec["H"] if H is None else H
            hidden = torch.randn((T, H), generator=g, device=device).to(torch.bfloat16)
            weight = (torch.randn((V, H), generator=g, device=device) * 0.02).to(torch.bfloat16)
            ids = torch.empty(T, dtype=torch.int64, device=device)
            lp_inf = torch.empty(T, dtype=torch.float32, device=device)
            for r0 in range(0, T, chunk_rows):
                r1 = min(T, r0 + chunk_rows)
                zc = hidden[r0:r1].float() @ weight.float().t()
                zi = zc + torch.randn(zc.shape, generator=g, device=device) * 0.15
                ids[r0:r1] = _gumbel_argmax(zi, g)
                lp_inf[r0:r1] = _engine_logprob(zi, ids[r0:r1])
            return Batch(cfg, T, V, None, ids.int(), lp_inf, adv, mask, cu, spec["lam"],
                         hidden=hidden, weight=weight)

        logits = torch.empty((T, V), dtype=torch.bfloat16, device=device)
        ids = torch.empty(T, dtype=torch.int64, device=device)
        lp_inf = torch.empty(T, dtype=torch.float32, device=device)
        lo, hi = math.log(1e-4), math.log(0.9999)
        pstar = torch.exp(lo + (hi - lo) * torch.rand(T, generator=g, device=device,
                                                      dtype=torch.float64)).float()
        spike = torch.zeros(T, dtype=torch.bool, device=device)
        infer = torch.empty((T, V), dtype=torch.bfloat16, device=device) if keep_infer else None
        if cfg == 4:
            valid = torch.nonzero(mask.cpu()).view(-1)
            n_sp = round(0.01 * valid.numel())
            spike[valid[torch.randperm(valid.numel(), generator=gcpu)[:n_sp]].to(device)] = True
        for r0 in range(0, T, chunk_rows):
            r1 = min(T, r0 + chunk_rows)
            z = _tempered_rows(r1 - r0, V, pstar[r0:r1], g, device).to(torch.bfloat16)
            logits[r0:r1] = z
            zi = z.float() + torch.randn((r1 - r0, V), generator=g, device=device) * 0.15
            y = _gumbel_argmax(zi, g)
            ids[r0:r1] = y
            sp = spike[r0:r1]
            if bool(sp.any()):
                rr = torch.nonzero(sp).view(-1)
                zi[rr, y[rr]] -= 6.0
            lp_inf[r0:r1] = _engine_logprob(zi, y)
            if infer is not None:
                infer[r0:r1] = zi.to(torch.bfloat16)
        extra = {"pstar": pstar, "spike": spike}
        if infer is not None:
            extra["logits_infer"] = infer
        return Batch(cfg, T, V, logits, ids.int(), lp_inf, adv, mask, cu, spec["lam"],
                     extra=extra)

    raise ValueError(f"unknown workload {cfg}")


def make_edge_rows(kind: str, V: int, T: int = 8, device="cpu", seed: int = 5,
                   dtype=torch.bfloat16) -> Batch:
    """Small hand-shaped batches for edge cases (all tokens valid unless stated).

    kinds: "neg_inf" (-inf logits except at the sampled token), "one_hot" (one
    logit far above the rest, p -> 1), "flat" (all logits equal), "ties" (the
    maximum shared by several entries), "huge" (|z| ~ 1e4), "nan" (a NaN in row
    1), "masked_half" (every other token masked)."""
    g = _gen(seed, device)
    z = torch.randn((T, V), generator=g, device=device) * 2.0
    ids = torch.randint(0, V, (T,), generator=g, device=device)
    mask = torch.ones(T, dtype=torch.uint8, device=device)
    if kind == "neg_inf":
        keep = torch.rand((T, V), generator=g, device=device) < 0.3
        z = torch.where(keep, z, torch.full_like(z, float("-inf")))
        z[torch.arange(T, device=device), ids] = 1.0
    elif kind == "one_hot":
        z[torch.arange(T, device=device), ids] = 60.0
    elif kind == "flat":
        z = torch.full_like(z, 0.75)
    elif kind == "ties":
        z[:, : max(1, V // 8)] = 9.0
    elif kind == "huge":
        z = z * 5000.0
    elif kind == "nan":
        z[1, V // 2] = float("nan")
    elif kind == "masked_half":
        mask[1::2] = 0
    else:
        raise ValueError(kind)
    zq = z.to(dtype)
    zi = zq.float().nan_to_num(nan=0.0) + torch.randn((T, V), generator=g, device=device) * 0.2
    lp_inf = _engine_logprob(zi, ids)
    lp_inf = torch.minimum(lp_inf, torch.full_like(lp_inf, -1e-7))
    adv = torch.randn(T, generator=g, device=device)
    cu = torch.tensor([0, T // 2, T], dtype=torch.int32, device=device)
    return Batch(0, T, V, zq.contiguous(), ids.int(), lp_inf.float(), adv.float(), mask, cu, 2.3)
