#!/usr/bin/env python3
"""Benchmark of the fused CIS token pass (forward + backward) on one GB300.

One step = one call of cis_loss_fwd_bwd over the whole batch: log-softmax of
the [T, V] bf16 training logits, the sampled-token log-probability, the CIS
weight (Algorithm 1), the PPO-clipped token loss (Eq. 1) and the bf16 gradient
with respect to the logits.  Workload: T = 16384 tokens (64 responses of 256,
groups of 8), V = 151936, temperatures spanning p in [1e-4, 0.9999]
(paper_2609_32444_gb300.synth, workload 3).  The logits (4.98 GB) are far
larger than the 129 MB L2, so no flush is needed between steps.

    python bench.py [--steps K] [--warmup W] [--gpus N] [--impl ours|reference]

Prints one JSON line (rank 0).  ``value`` is whole-job tokens/s with inputs
already in HBM; ``e2e`` is the same metric through the same C ABI with the
inputs in pinned host memory, copied in and the gradient copied out inside the
timed region.  ``--impl reference`` times the fp64 CPU oracle on the host
cores instead (a bounded sample of the same workload).
"""
import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "CIS loss fwd+bwd tokens/s at V=151936 bf16; achieved % of HBM roofline"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0
# the sources of each profiled kernel: a summary's traffic figure is used only
# while their hash matches the one recorded with it
FUSED_SOURCES = ["paper_2609_32444_gb300/csrc/cis_cluster.cu",
                 "paper_2609_32444_gb300/csrc/cis_dsmem.cuh",
                 "paper_2609_32444_gb300/csrc/cis_common.cuh"]
DIAG_SOURCES = ["paper_2609_32444_gb300/csrc/cis_diag.cu",
                "paper_2609_32444_gb300/csrc/cis_dsmem.cuh",
                "paper_2609_32444_gb300/csrc/cis_common.cuh"]
# committed ncu summaries that carry the full-size DRAM traffic per workload
PROFILE_SUMMARIES = {
    3: (os.path.join(ROOT, "profiles", "fused_pass_t16384_v151936_bf16.md"), FUSED_SOURCES),
    4: (os.path.join(ROOT, "profiles", "fused_pass_t65536_v151936_bf16_masked40.md"),
        FUSED_SOURCES),
    6: (os.path.join(ROOT, "profiles", "mismatch_t16384_v151936_bf16.md"), DIAG_SOURCES),
}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--mode", choices=["cis", "tis", "exact", "none"], default="cis")
    ap.add_argument("--workload", type=int, default=3, choices=[2, 3, 4, 5, 6])
    ap.add_argument("--dlogits", choices=["bf16", "f32"], default="bf16")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--e2e-chunk", type=int, default=512)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--tokens", type=int, default=None,
                    help="smaller T with the same recipe (for profiler captures only)")
    return ap.parse_args()


def dist_setup():
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "MEASURED_PEAKS.json hbm_gbs (measured copy bandwidth)"
    return FALLBACK_HBM_GBS, "fallback 6.8 TB/s (no MEASURED_PEAKS.json)"


def kernel_source_hash(sources=FUSED_SOURCES) -> str:
    h = hashlib.sha256()
    for rel in sources:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: int = 3, tokens=None):
    """DRAM bytes per launch of the main kernel from the committed ncu summary
    of this workload, if it was taken on the current kernel source (else None)."""
    entry = PROFILE_SUMMARIES.get(workload)
    if tokens is not None or entry is None or not os.path.exists(entry[0]):
        return None
    path, sources = entry
    txt = open(path).read()
    m = re.search(r"traffic_bytes_per_launch:\s*(\d+)", txt)
    s = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", txt)
    if not m or not s or s.group(1) != kernel_source_hash(sources):
        return None
    return int(m.group(1))


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.samples = []
        self.window = None
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(gpu_index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), line.strip()))

    def mark(self, t0, t1):
        self.window = (t0, t1)

    def summary(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        rows = [s for t, s in self.samples
                if self.window is None or self.window[0] <= t <= self.window[1] + 0.1]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            parts = [p.strip() for p in r.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


def physical_gpu_index(local_rank: int) -> int:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [v.strip() for v in vis.split(",") if v.strip()]
        if local_rank < len(ids) and ids[local_rank].isdigit():
            return int(ids[local_rank])
    return local_rank


def oracle_sample(batch_rows, mode, lam, seconds):
    """Time the fp64 oracle on host cores over repeated chunks of real rows."""
    import oracle
    import numpy as np
    logits, ids, lp, adv = batch_rows
    P = oracle.params(mode={"cis": 0, "tis": 1, "exact": 2, "none": 3}[mode], lam=lam)
    n = logits.shape[0]
    done, t0 = 0, time.perf_counter()
    while True:
        oracle.loss_fwd_bwd(logits, ids, lp, adv, P, rows=np.arange(n))
        done += n
        el = time.perf_counter() - t0
        if el >= seconds:
            return done, el


def host_rows(b, rows):
    import numpy as np
    import torch
    idx = torch.as_tensor(rows, device=b.logits.device)
    z = b.logits.index_select(0, idx).contiguous().cpu()
    z = z.view(torch.int16).numpy().view(np.uint16) if z.dtype == torch.bfloat16 else z.numpy()
    return (z, b.ids[idx].cpu().numpy(), b.lp_infer[idx].cpu().numpy(), b.adv[idx].cpu().numpy())


def run_reference(args, rank, world):
    """The reference arm: the fp64 oracle on the host cores, bounded samples."""
    if rank != 0:
        return
    import numpy as np
    import torch
    import oracle
    from paper_2609_32444_gb300 import synth
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    T_gen = None if dev == "cuda" else 256
    b = synth.make_batch(args.workload, device=dev, T=T_gen)
    spec = synth.WORKLOADS[args.workload]
    P = oracle.params(mode={"cis": 0, "tis": 1, "exact": 2, "none": 3}[args.mode], lam=b.lam)
    rng = np.random.default_rng(0)
    valid = np.nonzero(b.mask.cpu().numpy())[0]
    # size one step to about 0.1 s of oracle work
    probe = host_rows(b, rng.choice(valid, 16, replace=False))
    t0 = time.perf_counter()
    oracle.loss_fwd_bwd(*probe, P, rows=np.arange(16))
    per_row = (time.perf_counter() - t0) / 16
    nrows = int(max(8, min(len(valid), 0.1 / max(per_row, 1e-6))))
    sample = host_rows(b, rng.choice(valid, nrows, replace=False))
    for _ in range(args.warmup):
        oracle.loss_fwd_bwd(*sample, P, rows=np.arange(nrows))
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.loss_fwd_bwd(*sample, P, rows=np.arange(nrows))
    el = time.perf_counter() - t0
    value = nrows * args.steps / el
    cores = oracle.max_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": el / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": spec["name"], "T": spec["T"], "V": spec["V"], "mode": args.mode,
                   "lambda": b.lam, "kappa": 5e-3, "dlogits": "f64",
                   "sample_rows_per_step": nrows},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"{nrows} valid rows of {spec['name']} per step, fp64 "
                                   f"loss + weights + dlogits for every row"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args, rank, world, local):
    import numpy as np
    import torch
    from paper_2609_32444_gb300 import binding, build, synth

    build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    spec = synth.WORKLOADS[args.workload]
    b = synth.make_batch(args.workload, device=dev, seed=1000 + args.workload + 7919 * rank,
                         T=args.tokens)
    T, V = b.T, b.V
    dz_dt = torch.bfloat16 if args.dlogits == "bf16" else torch.float32
    P = binding.cis_default_params(args.mode, lam=b.lam)
    dz = torch.empty((T, V), dtype=dz_dt, device=dev)
    ws = torch.empty(binding.cis_loss_workspace_size(T, V), dtype=torch.uint8, device=dev)

    def step(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv, mask=b.mask):
        return binding.cis_loss_fwd_bwd(logits, ids, lp, adv, P, mask=mask, dlogits=dz,
                                        workspace=ws)

    for _ in range(max(3, args.warmup)):
        out = step()
    torch.cuda.synchronize()
    if binding.device_status(ws) != 0:
        raise RuntimeError(f"device status {binding.device_status(ws)} after warm-up")
    barrier(world)

    stream = torch.cuda.current_stream()
    kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    for a_, z_ in kev:  # torch creates the CUDA event on first record
        a_.record(stream)
        z_.record(stream)
    clocks = ClockSampler(physical_gpu_index(local))
    time.sleep(0.5)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    barrier(world)
    h0 = time.time()
    start.record(stream)
    for i in range(args.steps):
        binding.cis_profile_next_call(*kev[i])
        out = step()
    end.record(stream)
    torch.cuda.synchronize()
    h1 = time.time()
    barrier(world)
    clocks.mark(h0, h1)
    elapsed_ms = start.elapsed_time(end)
    kernel_ms = statistics.mean(a.elapsed_time(z) for a, z in kev)
    elapsed_ms = max_over_ranks(elapsed_ms, world)
    ms_per_step = elapsed_ms / args.steps
    value = T * world / (ms_per_step / 1e3)
    clk = clocks.summary()

    # ---- end to end through the C ABI with the batch in (pinned) host memory:
    # cis_loss_fwd_bwd_host streams the rows through the GPU in chunks
    e2e = None
    if args.e2e_steps > 0:
        hb = {k: v.cpu().contiguous().pin_memory() for k, v in
              dict(logits=b.logits, ids=b.ids, lp=b.lp_infer, adv=b.adv, mask=b.mask).items()}
        dz_h = torch.empty((T, V), dtype=dz_dt).pin_memory()
        hout = {}
        hws = torch.empty(binding.cis_loss_host_workspace_size(T, V, b.logits.dtype, dz_dt,
                                                               args.e2e_chunk),
                          dtype=torch.uint8, device=dev)

        def host_step():
            return binding.cis_loss_fwd_bwd_host(hb["logits"], hb["ids"], hb["lp"], hb["adv"], P,
                                                 dz_h, mask=hb["mask"],
                                                 chunk_tokens=args.e2e_chunk, workspace=hws,
                                                 outputs=hout)
        host_step()
        torch.cuda.synchronize()
        h2d = sum(v.numel() * v.element_size() for v in hb.values())
        d2h = dz_h.numel() * dz_h.element_size() + T * (4 + 4 + 1) + 8 + 48
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.e2e_steps):
            host_step()
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1), world) / args.e2e_steps
        e2e = {"value": T * world / (e2e_ms / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
               "api": f"cis_loss_fwd_bwd_host, chunks of {args.e2e_chunk} tokens",
               "link_GBps": (h2d + d2h) / (e2e_ms / 1e3) / 1e9}
        del hb, dz_h, hws

    # ---- roofline of the main kernel
    isz = b.logits.element_size()
    osz = dz.element_size()
    side = 4 + 4 + 4 + 1 + 4 + 4 + 4 + 1 + 4 + 1 + 4 + 8  # per-token inputs/outputs, bytes
    nvalid = int(b.mask.sum().item())
    alg_bytes = nvalid * V * isz + T * V * osz + T * side
    peak, peak_src = measured_peaks()
    achieved = alg_bytes / (kernel_ms / 1e3) / 1e9
    traffic = profiled_traffic(args.workload, args.tokens)
    # the library's layout: rows of 40-80 KB on two CTAs of 128 threads, the
    # rest on clusters of CTAs of 256 threads
    in_t = "bf16" if isz == 2 else "f32"
    out_t = "bf16" if osz == 2 else "f32"
    width = 128 if 40 * 1024 < V * isz <= 80 * 1024 else 256
    roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
            "frac": achieved / peak, "traffic": traffic,
            "kernel": f"cis_fused_cluster_kernel<{in_t},{out_t},{width}> "
                      "(fused fwd+bwd vocabulary pass)",
            "kernel_ms": kernel_ms, "algorithmic_bytes_per_launch": alg_bytes,
            "peak_source": peak_src, "frac_of_nominal_8000": achieved / NOMINAL_HBM_GBS,
            "step_frac": alg_bytes / (ms_per_step / 1e3) / 1e9 / peak}

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        rng = np.random.default_rng(0)
        valid = np.nonzero(b.mask.cpu().numpy())[0]
        rows = rng.choice(valid, min(256, len(valid)), replace=False)
        done, el = oracle_sample(host_rows(b, rows), args.mode, b.lam, args.cpu_seconds)
        import oracle
        cpu = {"value": done / el, "unit": "tokens/s", "cores": oracle.max_threads(),
               "kind": "oracle",
               "sample": f"{len(rows)} valid rows of {spec['name']} repeated for "
                         f"{el:.1f} s ({done} rows), fp64 loss + weights + dlogits"}

    st = binding.decode_stats(out["stats"])
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": spec["name"] if args.tokens is None else
                       f"{spec['name']} (T reduced to {T})", "T": T, "V": V, "mode": args.mode,
                       "lambda": b.lam, "kappa": 5e-3, "io_dtype": "bf16" if isz == 2 else "f32",
                       "dlogits": args.dlogits, "valid_tokens": nvalid,
                       "l2": "no flush: the 4.98 GB of logits per step exceed the 129 MB L2",
                       "parallelism": f"independent batch per GPU x{world}"},
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": 3 * args.steps,
            "clocks": clk,
            "check": {"loss": st["loss"], "n_truncated": st["n_truncated"],
                      "status": st["status"]},
        }
        print(json.dumps(line), flush=True)


def run_lmhead(args, rank, world, local):
    """Workload 5: the token pass fused with the LM head (tensor-core bound)."""
    import numpy as np
    import torch
    from paper_2609_32444_gb300 import binding, build, synth

    build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    spec = synth.WORKLOADS[5]
    b = synth.make_batch(5, device=dev, seed=1005 + 7919 * rank, T=args.tokens)
    T, V, H = b.T, b.V, b.hidden.shape[1]
    P = binding.cis_default_params(args.mode, lam=b.lam)
    nws = binding.cis_lmhead_workspace_size(T, V, H)
    wbuf = torch.empty(nws + 1024, dtype=torch.uint8, device=dev)
    ws = wbuf[(-wbuf.data_ptr()) % 1024:][:nws]
    # the library's default vocabulary chunk (dz of a chunk within 1 GiB)
    tp = -(-T // 128) * 128
    chunk = min(-(-V // 256) * 256, max(256, (1 << 30) // (2 * tp) // 256 * 256))
    n_chunks = -(-V // chunk)
    # scales, FWD, token, (DZ, then DH and DW in one launch) per chunk, reduce
    launches_per_call = 3 + 2 * n_chunks + 1

    def step():
        return binding.cis_lmhead_fused(b.hidden, b.weight, b.ids, b.lp_infer, b.adv, P,
                                        mask=b.mask, workspace=ws)

    for _ in range(max(3, args.warmup)):
        out = step()
    torch.cuda.synchronize()
    barrier(world)
    clocks = ClockSampler(physical_gpu_index(local))
    time.sleep(0.5)
    stream = torch.cuda.current_stream()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    h0 = time.time()
    start.record(stream)
    for _ in range(args.steps):
        out = step()
    end.record(stream)
    torch.cuda.synchronize()
    h1 = time.time()
    clocks.mark(h0, h1)
    ms = max_over_ranks(start.elapsed_time(end), world) / args.steps
    flops = 3 * 2.0 * T * V * H  # logits, dH, dW: the algorithmic work
    peaks = {}
    pp = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(pp):
        peaks = json.load(open(pp))
    peak = float(peaks.get("bf16_tflops_sustained", 1700.0))
    achieved = flops / (ms / 1e3) / 1e12
    st = binding.decode_stats(out["stats"])
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        import oracle
        rows = np.arange(0, T, max(1, T // 8))[:8]
        hb = b.hidden.cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        wb = b.weight.cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        t0 = time.perf_counter()
        oracle.lmhead_fwd_bwd(hb, wb, b.ids.cpu().numpy(), b.lp_infer.cpu().numpy(),
                              b.adv.cpu().numpy(), oracle.params(lam=b.lam), rows=rows,
                              n_valid_total=T, want_dw=False)
        el = time.perf_counter() - t0
        cpu = {"value": len(rows) / el, "unit": "tokens/s", "cores": oracle.max_threads(),
               "kind": "oracle",
               "sample": f"{len(rows)} tokens: fp64 logits over V={V}, weights, loss, dH rows "
                         f"(dW not included: it needs every token)"}
    if rank == 0:
        line = {
            "metric": "CIS fused LM-head fwd+bwd tokens/s at V=151936, H=2048 bf16",
            "value": T * world / (ms / 1e3), "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": spec["name"], "T": T, "V": V, "H": H, "mode": args.mode,
                       "grad_dtype": "f32", "vocab_chunk": chunk,
                       "l2": "operands (0.69 GB) exceed L2"},
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak,
                         "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
                         "algorithmic_flops": flops,
                         "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained",
                         "note": f"whole call ({launches_per_call} launches): logits, their "
                                 f"recomputation per vocabulary chunk ({n_chunks} chunks of "
                                 f"{chunk}), dH and dW on the tensor cores; the algorithmic "
                                 f"work counts the logits once"},
            "cpu_baseline": cpu, "e2e": None, "gpu_launches": launches_per_call * args.steps,
            "clocks": clocks.summary(),
            "check": {"loss": st["loss"], "status": st["status"]},
        }
        print(json.dumps(line), flush=True)


def run_diag(args, rank, world, local):
    """Workload 6: the mismatch diagnostics over both engines' logits."""
    import numpy as np
    import torch
    from paper_2609_32444_gb300 import binding, build, synth

    build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    spec = synth.WORKLOADS[6]
    b = synth.make_batch(6, device=dev, seed=1006 + 7919 * rank, T=args.tokens)
    T, V = b.T, b.V
    zi = b.extra["logits_infer"]
    P = binding.cis_default_params(args.mode, lam=b.lam)

    def step():
        return binding.cis_mismatch_diagnostics(b.logits, zi, b.ids, P, mask=b.mask)

    for _ in range(max(3, args.warmup)):
        out = step()
    torch.cuda.synchronize()
    barrier(world)
    stream = torch.cuda.current_stream()
    clocks = ClockSampler(physical_gpu_index(local))
    time.sleep(0.5)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    barrier(world)
    h0 = time.time()
    start.record(stream)
    for _ in range(args.steps):
        out = step()
    end.record(stream)
    torch.cuda.synchronize()
    h1 = time.time()
    barrier(world)
    clocks.mark(h0, h1)
    ms = max_over_ranks(start.elapsed_time(end), world) / args.steps
    # one launch per call: both tensors read once from HBM (the second pass
    # re-reads each row from L2), ids and mask read, five floats written per
    # position
    alg_bytes = 2 * T * V * b.logits.element_size() + T * (4 + 1) + 5 * 4 * T
    peak, peak_src = measured_peaks()
    achieved = alg_bytes / (ms / 1e3) / 1e9
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        import oracle
        rows = [0]
        zt_h = b.logits[rows].cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        zi_h = zi[rows].cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        t0 = time.perf_counter()
        oracle.mismatch_diagnostics(zt_h, zi_h, b.ids[rows].cpu().numpy(),
                                    oracle.params(mode={"cis": 0, "tis": 1, "exact": 2,
                                                        "none": 3}[args.mode], lam=b.lam))
        el = time.perf_counter() - t0
        cpu = {"value": len(rows) / el, "unit": "positions/s", "cores": 1, "kind": "oracle",
               "sample": f"{len(rows)} position of V={V} ({el:.0f} s): explicit fp64 "
                         f"expectation vectors (O(V^2) per position), one host thread; one "
                         f"position is the smallest sample"}
    if rank == 0:
        line = {
            "metric": "CIS mismatch diagnostics positions/s at V=151936 bf16 (two logit tensors)",
            "value": T * world / (ms / 1e3), "unit": "positions/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": spec["name"], "T": T, "V": V, "mode": args.mode,
                       "io_dtype": "bf16",
                       "l2": "no flush: the 9.96 GB of logits per step exceed the L2"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": profiled_traffic(6, args.tokens),
                         "kernel": "cis_mismatch_stream_kernel<cis, 16 warps, 1 CTA per SM> (both rows "
                                   "streamed through shared memory twice, HBM once)",
                         "algorithmic_bytes_per_launch": alg_bytes, "peak_source": peak_src},
            "cpu_baseline": cpu, "e2e": None, "gpu_launches": args.steps,
            "clocks": clocks.summary(),
        }
        print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    rank, world, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, rank, world)
    elif args.workload == 5:
        run_lmhead(args, rank, world, local)
    elif args.workload == 6:
        run_diag(args, rank, world, local)
    else:
        run_ours(args, rank, world, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
