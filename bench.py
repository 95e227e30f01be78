"""Benchmark of the SA sketching step (forward + backward) on one GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

One step = one pass of the whole hot path over the 100K-token training batch:
sa_sketch_fwd (saving the per-token lse) then sa_sketch_bwd, on 128 users x
100000 tokens, H=8 heads, d=128, P=512 prototypes, bf16 inputs with fp32
accumulation; K, V ~ N(0,1), Q ~ N(0, 0.02), dsketch ~ N(0,1), seeded.
Inputs (52 GB of K and V) are far larger than L2, so no flush is needed.

Prints ONE JSON line (rank 0).  `value` is sketched tokens/s of the whole job
(tokens = sum of user lengths; every head included).  Under torchrun each rank
runs its own full batch (weak scaling, no collective on the data path; the
timing is the max over ranks).  `--impl reference` times the fp64 CPU oracle
on a bounded sample of the same workload on the host cores instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_08443_gb300 import roofline as rf  # noqa: E402
from paper_2609_08443_gb300 import workloads as wl  # noqa: E402

METRIC = "SA sketched tokens/sec fwd and fwd+bwd at 100K/user; % of roofline"
CONFIG_ID = 4


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                "sm_max_mhz": d.get("sm_max_mhz", 2070.0), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0,
            "source": "fallback"}


def workload_config(spec, lens):
    return {"workload": "SA sketch training step (fwd+bwd), 100K tokens/user",
            "users": int(lens.size), "tokens_per_user": int(lens[0]), "tokens": int(lens.sum()),
            "heads": spec.H, "d": spec.d, "prototypes": spec.P, "inputs": "bf16 K,V,Q; fp32 accumulate",
            "l2": "inputs larger than L2 (K+V = %.1f GB per step), no flush" % (
                2 * lens.sum() * spec.H * spec.d * 2 / 1e9),
            "q_std": spec.q_std, "seed": spec.seed}


# ------------------------------------------------------------ clocks sampling

class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        fd, self.path = tempfile.mkstemp(prefix="sa_bench_clocks_", suffix=".csv")
        os.close(fd)

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()
        self.lines = open(self.path).read().splitlines() if os.path.exists(self.path) else []
        try:
            os.remove(self.path)
        except OSError:
            pass

    def summary(self):
        if self.proc is None or not self.lines:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "samples": len(sm),
                "reasons": sorted(reasons)}


# --------------------------------------------------------------- oracle timing

def oracle_sample(spec, budget_s=20.0, max_heads=None):
    """Time the fp64 oracle (fwd+bwd) on one user of the workload, head by head,
    until about ``budget_s`` of CPU work; returns tokens/s scaled to all heads."""
    from oracle import sa_backward, sa_forward

    L = int(wl.lengths(spec)[0])
    rng = np.random.default_rng(0)
    Q = (spec.q_std * rng.standard_normal((1, spec.P, spec.d))).astype(np.float32).astype(np.float64)
    cu = np.array([0, L])
    heads = 0
    t_tot = 0.0
    max_heads = max_heads or spec.H
    while heads < max_heads and (t_tot < budget_s or heads == 0):
        K = wl.bf16_bits_to_f64(wl.f32_to_bf16_bits(rng.standard_normal((L, 1, spec.d), dtype=np.float32)))
        V = wl.bf16_bits_to_f64(wl.f32_to_bf16_bits(rng.standard_normal((L, 1, spec.d), dtype=np.float32)))
        G = rng.standard_normal((1, 1, spec.P, spec.d))
        t0 = time.perf_counter()
        sa_forward(K, V, cu, Q, spec.scale, with_lse=True)
        sa_backward(K, V, cu, Q, spec.scale, G)
        t_tot += time.perf_counter() - t0
        heads += 1
    tokens_equiv = L * heads / spec.H
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {"value": tokens_equiv / t_tot, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"fp64 numpy oracle fwd+bwd on 1 user x {heads} of {spec.H} heads x {L} tokens "
                      f"(P={spec.P}, d={spec.d}); {t_tot:.1f} s; numpy/BLAS threads on {cores} host cores",
            "seconds": t_tot}


def run_reference(args, spec, lens):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    step_times = []
    info = None
    for s in range(args.warmup + args.steps):
        info = oracle_sample(spec, budget_s=0.0, max_heads=1)
        if s >= args.warmup:
            step_times.append(info["seconds"])
    t = sum(step_times)
    L = int(lens[0])
    tokens_equiv = L / spec.H * len(step_times)
    value = tokens_equiv / t
    cpu = {"value": value, "unit": "tokens/s", "cores": info["cores"], "kind": "oracle",
           "sample": f"each step: fp64 oracle fwd+bwd on 1 user x 1 of {spec.H} heads x {L} tokens"}
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * t / len(step_times), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": workload_config(spec, lens),
            "cpu_baseline": cpu,
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------- GPU arm

def job_rate(ms_local, tokens_per_rank, steps, world, device):
    """Whole-job timing of N ranks that each processed `tokens_per_rank` tokens
    per step for `steps` steps: the slowest rank's time (all-reduce MAX; each
    rank is an independent replica, so this is the only collective) and the
    job's tokens/s over it.  Returns (ms, tokens/s), the same on every rank."""
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(ms_local)], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    ms = float(t.item())
    return ms, tokens_per_rank * world * steps / (ms / 1e3)


def run_ours(args, spec, lens):
    import torch
    import torch.distributed as dist

    from paper_2609_08443_gb300 import binding

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    binding.load()
    pk = peaks()

    data = wl.make_device(spec, dev)
    K, V, Q, cu, dS = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    B = int(lens.size)
    N, H, d = K.shape
    P = Q.shape[1]
    tokens = int(lens.sum())
    sketch = torch.empty((B, H, P, d), dtype=torch.float32, device=dev)
    lse = torch.empty((N, H), dtype=torch.float32, device=dev)
    dK, dV = torch.empty_like(K), torch.empty_like(V)
    dQ = torch.empty((H, P, d), dtype=torch.float32, device=dev)
    ws = torch.empty(binding.sa_workspace_size(B, N, H, P, d, binding.SA_BF16, 1), dtype=torch.uint8, device=dev)

    def step():
        binding.sa_sketch_fwd(K, V, cu, Q, spec.scale, out=sketch, lse_out=lse, ws=ws)
        binding.sa_sketch_bwd(K, V, cu, Q, dS, spec.scale, lse=lse, outs=(dK, dV, dQ), ws=ws)

    for _ in range(args.warmup):
        step()
    if binding.sa_get_device_error(ws) != 0:
        raise RuntimeError("device-side error during warm-up")

    # fwd-only timing (same inputs), for the forward half of the metric
    stream = torch.cuda.current_stream(dev)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(max(1, args.steps)):
        binding.sa_sketch_fwd(K, V, cu, Q, spec.scale, out=sketch, lse_out=lse, ws=ws)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    fwd_ms = e0.elapsed_time(e1) / max(1, args.steps)

    # timed region: K steps, barrier + synchronize on both sides, kernel events on
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    binding.sa_timing_enable(True)
    n_launch0 = binding.sa_launch_count()
    with Clocks(local) as clk:
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize(dev)
    launches = binding.sa_launch_count() - n_launch0
    ms = e0.elapsed_time(e1)
    fwd_k_ms, fwd_k_n = binding.sa_timing_read(binding.SA_KERNEL_FWD_MAIN)
    bwd_k_ms, bwd_k_n = binding.sa_timing_read(binding.SA_KERNEL_BWD_MAIN)
    per_kernel = {}
    for cls, label in ((binding.SA_KERNEL_FWD_LSE, "fwd_lse"), (binding.SA_KERNEL_FWD_MAIN, "fwd_main"),
                       (binding.SA_KERNEL_BWD_MAIN, "bwd_main"), (binding.SA_KERNEL_BWD_DQ, "bwd_dq")):
        kms, kn = binding.sa_timing_read(cls)
        if kn:
            per_kernel[label] = {"ms_per_call": kms / args.steps, "launches": kn}
    # the backward's main kernels: token side plus prototype-side dQ when split
    if "bwd_dq" in per_kernel:
        bwd_k_ms += per_kernel["bwd_dq"]["ms_per_call"] * args.steps
        bwd_k_n += per_kernel["bwd_dq"]["launches"]
    binding.sa_timing_enable(False)
    if binding.sa_get_device_error(ws) != 0:
        raise RuntimeError("device-side error in the timed region")
    ms, value = job_rate(ms, tokens, args.steps, world, dev)
    ms_per_step = ms / args.steps

    # roofline of the dominant kernel (the backward main kernel) and of the forward
    eb = 2
    fw = rf.fwd_work(tokens, B, H, P, d, eb, lse=True)
    bw = rf.bwd_work(tokens, B, H, P, d, eb, lse_in=True)
    peak_t = pk["bf16_tflops_sustained"]

    def roof(work, kms, kn, name, calls):
        """Achieved rate of a call's main kernels: algorithmic work of one call
        divided by the summed device time of its main-kernel launches."""
        if kn == 0:
            return None
        per_call_s = kms / calls / 1e3
        t_tensor = work.flops / (peak_t * 1e12)
        t_hbm = work.bytes / (pk["hbm_gbs"] * 1e9)
        if t_tensor >= t_hbm:
            ach, peak, unit, bound = work.flops / per_call_s / 1e12, peak_t, "TFLOP/s", "tensor"
        else:
            ach, peak, unit, bound = work.bytes / per_call_s / 1e9, pk["hbm_gbs"], "GB/s", "hbm"
        return {"kernel": name, "bound": bound, "achieved": ach, "peak": peak, "unit": unit, "frac": ach / peak,
                "traffic": traffic_for(name), "traffic_per": "call (DRAM bytes, ncu, scaled from a sub-batch)",
                "avg_launch_ms": kms / kn, "launches": kn,
                "launches_per_call": kn // calls, "ms_per_call": kms / calls,
                "peak_source": f"{pk['source']} ({'bf16 sustained' if unit == 'TFLOP/s' else 'HBM copy'})",
                "algorithmic_per_call": work.flops if unit == "TFLOP/s" else work.bytes}

    bwd_name = binding.sa_main_kernel_name(P, d, binding.SA_BF16, True)
    fwd_name = binding.sa_main_kernel_name(P, d, binding.SA_BF16, False)
    r_bwd = roof(bw, bwd_k_ms, bwd_k_n, bwd_name, args.steps)
    r_fwd = roof(fw, fwd_k_ms, fwd_k_n, fwd_name, args.steps)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    exp_ps = rf.exp_peak_per_s(sms, pk["sm_max_mhz"])
    step_w = rf.step_work(tokens, B, H, P, d, eb)
    t_roof = rf.roofline_time(step_w, peak_t, pk["hbm_gbs"], exp_ps)
    t_roof_fwd = rf.roofline_time(fw, peak_t, pk["hbm_gbs"], exp_ps)

    tw = tokenwise_leg(args, spec, data, dev, pk) if rank == 0 else None
    e2e = e2e_run(args, spec, data, (dK, dV), dev) if rank == 0 else None
    # the other workloads, after the 100K batch's buffers are released
    del data, K, V, Q, cu, dS, sketch, lse, dK, dV, dQ, ws
    torch.cuda.empty_cache()
    others = {f"config{i}": config_leg(i, args, dev, pk, exp_ps) for i in (1, 2, 3, 5)} if rank == 0 else None
    cpu = oracle_sample(spec, budget_s=15.0) if (rank == 0 and world == 1) else None

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": workload_config(spec, lens),
                "fwd": {"value": tokens * world / (fwd_ms / 1e3), "unit": "tokens/s", "ms_per_call": fwd_ms,
                        "roofline_bound": t_roof_fwd["bound"], "roofline_ms": t_roof_fwd["time"] * 1e3,
                        "roofline_frac": (t_roof_fwd["time"] * 1e3) / fwd_ms},
                "step_roofline": {"bound": t_roof["bound"], "ms": t_roof["time"] * 1e3,
                                  "frac": t_roof["time"] * 1e3 / ms_per_step,
                                  "terms_ms": {k: t_roof[k] * 1e3 for k in ("tensor", "hbm", "mufu")}},
                "mufu_peak": {"ex2_per_s": exp_ps, "per_sm_clk": rf.EX2_PER_SM_CLK, "sms": sms,
                              "sm_mhz": pk["sm_max_mhz"], "source": "ex2.approx throughput probe (measured)"},
                "roofline": r_bwd, "roofline_fwd": r_fwd,
                "cpu_baseline": cpu, "e2e": e2e, "clocks": clk.summary(), "gpu_launches": int(launches),
                "kernels": {"fwd": fwd_name, "bwd": bwd_name}, "kernel_ms": per_kernel, "tokenwise": tw,
                "workloads": others}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def config_leg(cfg, args, dev, pk, exp_ps):
    """One of the other evaluation workloads at full size through the C ABI:
    the forward alone and, where the workload trains, forward (saving lse) +
    backward, each timed over K calls with CUDA events after warm-up, against
    its roofline (slowest of tensor FLOPs, HBM bytes and exp2 at their peaks).
    Reported beside the headline, not part of it."""
    import torch

    from paper_2609_08443_gb300 import binding

    spec = wl.config(cfg)
    lens = wl.lengths(spec)
    data = wl.make_device(spec, dev)
    K, V, Q, cu, dS = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    B = int(lens.size)
    N, H, d = K.shape
    P = Q.shape[1]
    tokens = int(lens.sum())
    code = binding.SA_BF16 if K.dtype == torch.bfloat16 else binding.SA_F32
    eb = K.element_size()
    sketch = torch.empty((B, H, P, d), dtype=torch.float32, device=dev)
    lse = torch.empty((N, H), dtype=torch.float32, device=dev)
    ws = torch.empty(binding.sa_workspace_size(B, N, H, P, d, code, int(spec.bwd)), dtype=torch.uint8, device=dev)
    outs = (torch.empty_like(K), torch.empty_like(V), torch.empty((H, P, d), dtype=torch.float32, device=dev))
    stream = torch.cuda.current_stream(dev)
    # small workloads: more calls per timing so the events cover well over a millisecond
    reps = max(args.steps, 20)

    def timed(fn):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / reps

    def fwd():
        binding.sa_sketch_fwd(K, V, cu, Q, spec.scale, out=sketch, lse_out=lse, ws=ws)

    def step():
        fwd()
        binding.sa_sketch_bwd(K, V, cu, Q, dS, spec.scale, lse=lse, outs=outs, ws=ws)

    # fp32 inputs run on the CUDA cores: their compute term is the FP32 FMA rate
    # (128 lanes x 2 FLOP per SM and clock), not the bf16 tensor peak
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    peak_c = pk["bf16_tflops"] if code == binding.SA_BF16 else sms * 128 * 2 * pk["sm_max_mhz"] * 1e6 / 1e12
    cname = "tensor" if code == binding.SA_BF16 else "fp32_fma"

    def entry(ms, work):
        r = rf.roofline_time(work, peak_c, pk["hbm_gbs"], exp_ps)
        bound = cname if r["bound"] == "tensor" else r["bound"]
        return {"ms": ms, "tokens_per_s": tokens / (ms / 1e3), "roofline_bound": bound,
                "roofline_ms": r["time"] * 1e3, "roofline_frac": r["time"] * 1e3 / ms,
                "terms_ms": {cname: r["tensor"] * 1e3, "hbm": r["hbm"] * 1e3, "mufu": r["mufu"] * 1e3}}

    out = {"workload": spec.name, "users": B, "tokens": tokens, "heads": H, "d": d, "prototypes": P,
           "dtype": "bf16" if code == binding.SA_BF16 else "f32",
           "kernels": {"fwd": binding.sa_main_kernel_name(P, d, code, False)},
           "tile_fill": tokens / (128.0 * int(np.sum((lens + 127) // 128))),
           "timing": f"CUDA events over {reps} calls after {args.warmup} warm-up calls; peaks: bf16 burst, HBM copy, "
                     "MUFU ex2 (measured)"}
    out["fwd"] = entry(timed(fwd), rf.fwd_work(tokens, B, H, P, d, eb, lse=True))
    if spec.bwd:
        out["kernels"]["bwd"] = binding.sa_main_kernel_name(P, d, code, True)
        out["fwd_bwd"] = entry(timed(step), rf.step_work(tokens, B, H, P, d, eb))
    if binding.sa_get_device_error(ws) != 0:
        raise RuntimeError(f"device-side error in workload {cfg}")
    del data, K, V, ws, outs
    torch.cuda.empty_cache()
    return out


def tokenwise_leg(args, spec, data, dev, pk):
    """The token-wise normalisation of Sec. 5.1 (weights normalised over each
    user's tokens) on the same inputs: K fwd+bwd steps through the C ABI, timed
    like the main step, with its main kernels' rates against the bf16 peak.
    Reported beside the headline, not part of it."""
    import torch

    from paper_2609_08443_gb300 import binding

    K, V, Q, cu, dS = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    B = cu.numel() - 1
    N, H, d = K.shape
    P = Q.shape[1]
    tokens = N
    lib = binding.load()
    ws = torch.empty(lib.sa_workspace_size_tokenwise(B, N, H, P, d, binding.SA_BF16, 1), dtype=torch.uint8,
                     device=dev)

    def step():
        O, lse = binding.sa_sketch_fwd_tokenwise(K, V, cu, Q, spec.scale, want_lse=True, ws=ws)
        return binding.sa_sketch_bwd_tokenwise(K, V, cu, Q, dS, spec.scale, sketch=O, lse=lse, ws=ws)

    for _ in range(max(1, args.warmup)):
        step()
    stream = torch.cuda.current_stream(dev)
    torch.cuda.synchronize(dev)
    binding.sa_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / args.steps
    kms = {}
    for cls, label in ((binding.SA_KERNEL_FWD_MAIN, "fwd_main"), (binding.SA_KERNEL_BWD_MAIN, "bwd_main"),
                       (binding.SA_KERNEL_BWD_DQ, "bwd_dq")):
        t, n = binding.sa_timing_read(cls)
        kms[label] = {"ms_per_call": t / args.steps, "launches": n}
    binding.sa_timing_enable(False)
    if binding.sa_get_device_error(ws) != 0:
        raise RuntimeError("device-side error in the token-wise leg")
    peak_t = pk["bf16_tflops_sustained"]
    fw = rf.fwd_work(tokens, B, H, P, d, 2, lse=True)
    bw = rf.bwd_work(tokens, B, H, P, d, 2, lse_in=True)
    f_ms = kms["fwd_main"]["ms_per_call"]
    b_ms = kms["bwd_main"]["ms_per_call"] + kms["bwd_dq"]["ms_per_call"]
    return {"value": tokens / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms, "kernel_ms": kms,
            "fwd_tflops": fw.flops / (f_ms / 1e3) / 1e12, "fwd_frac": fw.flops / (f_ms / 1e3) / 1e12 / peak_t,
            "bwd_tflops": bw.flops / (b_ms / 1e3) / 1e12, "bwd_frac": bw.flops / (b_ms / 1e3) / 1e12 / peak_t,
            "peak": peak_t, "peak_source": f"{pk['source']} (bf16 sustained)"}


def traffic_for(kernel_name):
    """DRAM bytes per call of the kernel (for the split backward: its token-side
    and dQ kernels together) from the committed ncu summary, if it matches the
    kernel source that is built now; else None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    try:
        d = json.load(open(p))
    except ValueError:
        return None
    ent = d.get(kernel_name)
    if not ent:
        return None
    from paper_2609_08443_gb300 import build

    return ent.get("bytes_per_call") if ent.get("source_hash") == build.source_hash() else None


def _meminfo_available():
    try:
        for line in open("/proc/meminfo"):
            if line.startswith("MemAvailable:"):
                return int(line.split()[1]) * 1024
    except OSError:
        pass
    return None


def copy_ceiling(h_src, h_dst, d_buf, dev, nbytes):
    """Plain page-locked copies of ``nbytes``: host-to-device alone,
    device-to-host alone, and both at once on two streams (GB/s, CUDA events)."""
    import torch

    n = nbytes // h_src.element_size()
    hs, hd, db = h_src.view(-1)[:n], h_dst.view(-1)[:n], d_buf.view(-1)
    dbi, dbo = db[:n], db[n:2 * n]
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def run(h2d, d2h):
        torch.cuda.synchronize(dev)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        ev[0].record(s1)
        s2.wait_event(ev[0])
        if h2d:
            with torch.cuda.stream(s1):
                dbi.copy_(hs, non_blocking=True)
        if d2h:
            with torch.cuda.stream(s2):
                hd.copy_(dbo, non_blocking=True)
        ev[1].record(s1)
        ev[2].record(s2)
        torch.cuda.synchronize(dev)
        ms = max(ev[0].elapsed_time(ev[1]), ev[0].elapsed_time(ev[2]))
        return (int(h2d) + int(d2h)) * nbytes / (ms / 1e3) / 1e9

    run(True, True)  # warm
    return {"h2d_gbs": max(run(True, False) for _ in range(3)), "d2h_gbs": max(run(False, True) for _ in range(3)),
            "both_gbs": max(run(True, True) for _ in range(3)), "bytes_each": int(nbytes),
            "how": "torch copy_ between page-locked host and device memory, CUDA events, best of 3"}


def array_copy_pass(ins, outs, dev, piece=1 << 30):
    """One plain pass of a step's copies over the very host arrays the e2e leg
    hands the library: every byte of ``ins`` host-to-device and every byte of
    ``outs`` device-to-host, the two directions at once on two streams, in
    pieces of ``piece`` bytes through two device buffers, no kernels.  Its rate
    is the copy ceiling of the step's pipeline on this host memory; on a GB300
    host it fell below the 4 GiB ceiling for ~100 GB of arrays after other
    processes had run.  Best of two passes, CUDA events."""
    import torch

    bufs = (torch.empty(piece, dtype=torch.uint8, device=dev), torch.empty(piece, dtype=torch.uint8, device=dev))
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def pieces(t):
        f = t.reshape(-1).view(torch.uint8)
        return [f[o:o + piece] for o in range(0, f.numel(), piece)]

    src = [p for t in ins for p in pieces(t)]
    dst = [p for t in outs for p in pieces(t)]
    nbytes = sum(p.numel() for p in src + dst)

    def run():
        torch.cuda.synchronize(dev)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        ev[0].record(s_in)
        s_out.wait_event(ev[0])
        with torch.cuda.stream(s_in):
            for p in src:
                bufs[0][:p.numel()].copy_(p, non_blocking=True)
        with torch.cuda.stream(s_out):
            for p in dst:
                p.copy_(bufs[1][:p.numel()], non_blocking=True)
        ev[1].record(s_in)
        ev[2].record(s_out)
        torch.cuda.synchronize(dev)
        return max(ev[0].elapsed_time(ev[1]), ev[0].elapsed_time(ev[2]))

    ms = min(run() for _ in range(2))
    return {"gbs": nbytes / (ms / 1e3) / 1e9, "ms": ms, "bytes": int(nbytes),
            "how": "the e2e arrays copied once in and once out (1 GiB pieces, two streams), no kernels, best of 2"}


class HostArrays:
    """Page-locked host arrays for the e2e leg: anonymous memory advised onto
    transparent huge pages (MADV_HUGEPAGE), touched, then registered with
    cudaHostRegister.  On a GB300 host, page-locked memory on small pages
    copied at 64-80 GB/s in some passes after other processes had run (a
    translation cost per page), against 193-211 GB/s on huge pages in the same
    state.  Falls back to torch's page-locked allocator where the mapping or the
    advice is refused."""

    def __init__(self):
        self.maps, self.regs, self.kind = [], [], "thp+cudaHostRegister"

    def empty(self, shape, dtype):
        import mmap

        import torch

        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        try:
            mm = mmap.mmap(-1, max(n, 1), flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
            mm.madvise(mmap.MADV_HUGEPAGE)
            t = torch.frombuffer(mm, dtype=torch.uint8, count=n).view(dtype).view(shape)
            t.zero_()  # fault the pages in (huge pages where the kernel grants them)
            if torch.cuda.cudart().cudaHostRegister(t.data_ptr(), n, 0) != 0:
                raise OSError("cudaHostRegister failed")
        except (OSError, ValueError, AttributeError):
            self.kind = "torch pin_memory"
            return torch.empty(shape, dtype=dtype, pin_memory=True)
        self.maps.append(mm)
        self.regs.append(t)
        return t

    @staticmethod
    def anon_huge_bytes():
        """This process's anonymous memory on transparent huge pages (bytes), or None."""
        try:
            with open("/proc/self/smaps_rollup") as fh:
                for line in fh:
                    if line.startswith("AnonHugePages:"):
                        return int(line.split()[1]) * 1024
        except OSError:
            pass
        return None

    def release(self):
        import torch

        torch.cuda.synchronize()
        for t in self.regs:
            torch.cuda.cudart().cudaHostUnregister(t.data_ptr())
        self.regs.clear()
        self.maps.clear()  # the mappings close once the tensors over them are gone


def e2e_run(args, spec, data, dkdv, dev):
    """Same metric through the public API with host buffers: every step hands the
    library page-locked host arrays (K, V, Q, dsketch) and gets the host arrays
    (sketch, dK, dV, dQ) back, through sa_sketch_step_host, which copies chunks of
    users in and out on its own streams while the step runs on the previous
    chunk.  Wall clock from the call to the synchronised results, every user of
    the workload unless the host lacks the page-locked memory for them."""
    import torch

    from paper_2609_08443_gb300 import binding

    lens = wl.lengths(spec)
    B_all, H, P, d = spec.B, spec.H, spec.P, spec.d

    def pinned_need(b):
        # K, V in and dK, dV out (bf16), dsketch in and sketch out (fp32); with the
        # fallback allocator each block is rounded up to a power of two
        n = int(lens[:b].sum())
        sizes = [n * H * d * 2] * 4 + [b * H * P * d * 4] * 2
        return sum(1 << (max(s, 1) - 1).bit_length() for s in sizes)

    avail = _meminfo_available()
    B = B_all
    while avail is not None and B > 1 and pinned_need(B) > 0.85 * avail:
        B -= 1
    N = int(lens[:B].sum())
    cu = torch.from_numpy(wl.cu_seqlens(lens[:B]))
    ha = HostArrays()
    huge0 = HostArrays.anon_huge_bytes()
    bf = torch.bfloat16
    h = {"K": ha.empty((N, H, d), bf), "V": ha.empty((N, H, d), bf), "Q": torch.empty((H, P, d), dtype=bf,
                                                                                     pin_memory=True),
         "dsketch": ha.empty((B, H, P, d), torch.float32), "cu_seqlens": cu.pin_memory()}
    for k in ("K", "V"):
        h[k].copy_(data[k][:N])
    h["Q"].copy_(data["Q"])
    h["dsketch"].copy_(data["dsketch"][:B])
    outs = (ha.empty((B, H, P, d), torch.float32), ha.empty((N, H, d), bf), ha.empty((N, H, d), bf),
            torch.empty((H, P, d), dtype=torch.float32, pin_memory=True))
    huge1 = HostArrays.anon_huge_bytes()
    ceiling = copy_ceiling(h["K"], outs[1], dkdv[0], dev, min(4 << 30, h["K"].numel() * 2 // 2))
    lib = binding.load()
    ws = torch.empty(lib.sa_step_host_workspace_size(h["cu_seqlens"].data_ptr(), B, H, P, d, binding.SA_BF16, 0),
                     dtype=torch.uint8, device=dev)
    h2d = sum(h[k].numel() * h[k].element_size() for k in ("K", "V", "Q", "dsketch", "cu_seqlens"))
    d2h = sum(o.numel() * o.element_size() for o in outs)

    def step():
        binding.sa_sketch_step_host(h["K"], h["V"], h["cu_seqlens"], h["Q"], h["dsketch"], spec.scale, outs=outs,
                                    device=dev, ws=ws)

    for _ in range(3):
        step()
    if binding.sa_get_device_error(ws) != 0:
        raise RuntimeError("device-side error in the e2e leg")
    n = max(3, min(args.steps, 7))
    times = []
    for _ in range(n):
        t0 = time.perf_counter()
        step()
        times.append(time.perf_counter() - t0)
    mean = sum(times) / len(times)
    med = statistics.median(times)
    arrays = array_copy_pass([h[k] for k in ("K", "V", "Q", "dsketch")], list(outs), dev)
    kind = ha.kind
    del h, outs
    ha.release()
    return {"value": N / mean, "unit": "tokens/s", "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "host_memory": kind,
            "host_huge_page_bytes": (huge1 - huge0) if huge0 is not None and huge1 is not None else None,
            "sample": f"{B} of the {B_all} users (same shapes), page-locked host arrays in and out through "
                      "sa_sketch_step_host (chunks of 262144 tokens, copies overlapped with the step), wall clock, "
                      f"mean of {n} steps" + ("" if B == B_all else
                                              f"; host MemAvailable {avail / 2**30:.0f} GiB limits the users"),
            "ms_per_step": mean * 1e3, "ms_per_step_median": med * 1e3, "value_median": N / med,
            "ms_per_step_all": [t * 1e3 for t in times],
            "copy_gbs": (h2d + d2h) / mean / 1e9, "copy_ceiling": ceiling, "array_copy": arrays}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    spec = wl.config(CONFIG_ID)
    lens = wl.lengths(spec)
    if args.impl == "reference":
        run_reference(args, spec, lens)
    else:
        run_ours(args, spec, lens)


if __name__ == "__main__":
    main()
