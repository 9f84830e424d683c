#!/usr/bin/env python
"""Throughput of K-interval attention forward + backward on GB300.

One step = kint_attn_fwd + kint_attn_bwd over one batch of the GPT-2-small
attention layer (B=8, H=12, T=1024, d=64, causal; K=4, FWM tau=8, Nearest,
Prob-STE, full calibration gradient; TF32 tensor products), inputs resident in
HBM.  The metric is algorithmic TFLOP/s: 6 causal T x T x d contractions per
step (QK^T, PV, dP, dV, dQ, dK), 6 * B*H*d*T*(T+1) flops.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl cuda|reference]

With N > 1 (launched by torch.distributed.run) every rank runs its own replica
of the workload on its own GPU (the operator shards over (b, h) with no
exchange); the value is the work of all ranks over the slowest rank's time.
``--impl reference`` times the fp64 CPU oracle on the host cores instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "K-interval attn fwd+bwd TFLOP/s @GPT-2-small shape; % of TF32 tensor peak"
UNIT = "TFLOP/s"
SHAPE = dict(B=8, H=12, T=1024, d=64)
VARIANT = dict(Kint=4, calib=1, tau=8.0, recon=1, ste=1, grad=0)  # FWM tau=8, Nearest, Prob-STE, full
WORKLOAD = ("GPT-2-small attention layer: B=8, H=12, T=1024, d_head=64, causal; K=4, FWM tau=8, Nearest, "
            "Prob-STE, full calibration gradients; fwd+bwd")
N_INPUT_SETS = 3  # rotated so that no step reads inputs the previous step left in L2
TF32_PER_BF16 = 1.1 / 2.25  # nominal dense TF32 : BF16 tensor rate of GB300 (1.1 : 2.25 PFLOP/s)


# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of each kernel from
# one ncu capture of this workload (profiles/traffic_gpt2_tf32.md), valid only for the
# kernel sources they were taken from.
TRAFFIC = {"src": "893f13747009898a", "k_prep": 65120486, "k_fwd_stats": 50400448, "k_fwd_main": 91583501,
           "k_bwd_fused": 378647168, "k_bwd_ext": 73677402}


def kernel_source_digest() -> str:
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_33591_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def unit_flops(B, H, T, d):
    """One causal T x T x d contraction over all heads: 2 * B*H*d*T(T+1)/2 flops."""
    return B * H * d * T * (T + 1)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            m = json.load(f)
        return {"hbm_gbs": float(m["hbm_gbs"]), "bf16": float(m["bf16_tflops"]),
                "bf16_sustained": float(m.get("bf16_tflops_sustained", m["bf16_tflops"])), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = max(mx, float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"samples": 0}
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        import torch
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return world, rank, local


def reduce_max(ms: float, world: int, device) -> float:
    """The slowest rank's time: every rank contributes its own, all receive the max."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(flops_per_step: float, world: int, ms: float) -> float:
    """Whole-job throughput: the work of all ranks (replicas) over the slowest rank's time."""
    return world * flops_per_step / (ms * 1e-3) / 1e12


def cpu_oracle_rate(n_heads: int, min_seconds: float = 0.0):
    """Time the fp64 oracle (fwd + bwd) on the first n_heads (b, h) heads of the
    workload at full length; return (TFLOP/s of algorithmic work, seconds, threads)."""
    import numpy as np
    import oracle
    from paper_2609_33591_gb300.inputs import make_qkvdo
    B, H, T, d = SHAPE["B"], SHAPE["H"], SHAPE["T"], SHAPE["d"]
    Q, K, V, dO = make_qkvdo(B, H, T, d, seed=1)
    sl = lambda X: np.ascontiguousarray(X.reshape(B * H, T, d)[:n_heads].reshape(1, n_heads, T, d))
    q, k, v, do = sl(Q), sl(K), sl(V), sl(dO)
    cfg = oracle.Config(**VARIANT)
    threads = min(oracle.hardware_threads(), n_heads)
    reps = 0
    t0 = time.perf_counter()
    while True:
        oracle.forward(q, k, v, cfg, lerp_out=True, nthreads=threads)
        oracle.backward(q, k, v, do, cfg, nthreads=threads)
        reps += 1
        dt = time.perf_counter() - t0
        if dt >= min_seconds:
            break
    return reps * 6 * unit_flops(1, n_heads, T, d) / dt / 1e12, dt, threads, reps


def bench_parity(Q, K, V, dO):
    """The timed workload's outputs against the fp64 oracle (outside the timed region, in
    the CPU-baseline leg): decisions, flip fraction, normwise errors, zero-sum residual."""
    from paper_2609_33591_gb300 import kint
    from tests import parity
    cfg = kint.Config(**VARIANT)
    rep, err = {}, None
    t0 = time.perf_counter()
    try:
        parity.check(Q, K, V, dO, cfg, kint.PREC_TF32, heads_per_chunk=12, report=rep, case="bench")
    except AssertionError as e:
        err = str(e)[:400]
    keys = ("flip_fraction", "bins_flips", "ivals_flips", "valid", "arg_max_flips", "errors", "p99_rel",
            "zero_sum_gpu", "zero_sum_oracle", "band")
    out = {"passed": err is None, "tol": parity.TOL[kint.PREC_TF32], "prec": "tf32",
           "oracle": "fp64 CPU oracle on the whole workload, 12 heads per chunk, decision-aligned",
           "seconds": time.perf_counter() - t0, **{k: rep.get(k) for k in keys}}
    if err:
        out["failure"] = err
    return out


def cublas_tf32_tflops(dev, n=8192, reps=10):
    """cuBLAS fp32 GEMM with TF32 tensor cores, n^3, best of `reps` (a measured TF32 peak on
    this GPU, beside the nominal-ratio one)."""
    import torch
    old = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = True
    try:
        a = torch.randn(n, n, device=dev)
        b = torch.randn(n, n, device=dev)
        c = torch.empty(n, n, device=dev)
        for _ in range(3):
            torch.matmul(a, b, out=c)
        best = float("inf")
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            torch.matmul(a, b, out=c)
            e1.record()
            torch.cuda.synchronize()
            best = min(best, e0.elapsed_time(e1))
        del a, b, c
        return 2.0 * n ** 3 / (best * 1e-3) / 1e12
    finally:
        torch.backends.cuda.matmul.allow_tf32 = old


# The other single-GPU workloads of the benchmark's configurations, timed like the headline
# (inputs larger than L2, CUDA events, warm-up first): name -> shape, seed, peaked-row
# fraction, operator, and whether the softmax comparator runs beside it.
OTHER_CONFIGS = {
    "1b_scale": dict(shape=(4, 16, 2048, 128), seed=3, peaked=0.05, softmax=False,
                     variant=dict(Kint=4, calib=1, tau=8.0, recon=1, ste=0, grad=0),
                     workload="1B-scale attention: B=4, H=16, T=2048, d=128, 5% peaked rows (+12 score); K=4, "
                              "FWM tau=8, Nearest, Weight-STE, full; TF32"),
    "long_context": dict(shape=(1, 16, 16384, 128), seed=4, peaked=0.0, softmax=True,
                         variant=dict(Kint=16, calib=0, tau=8.0, recon=0, ste=1, grad=0),
                         workload="long context: B=1, H=16, T=16384, d=128; K=16, MinMax, LERP, Prob-STE, full; "
                                  "TF32"),
}


def run_reference(args, world, rank):
    """The oracle as the reference arm, on a bounded sample per step."""
    if rank != 0:
        return 0
    heads = 16
    for _ in range(args.warmup):
        cpu_oracle_rate(heads)
    total_f, total_t, threads = 0.0, 0.0, 1
    for _ in range(args.steps):
        _, dt, threads, _ = cpu_oracle_rate(heads)
        total_t += dt
        total_f += 6 * unit_flops(1, heads, SHAPE["T"], SHAPE["d"])
    value = total_f / total_t / 1e12
    sample = f"{heads} of 96 (b,h) heads at T=1024 per step (fwd+bwd, fp64 oracle)"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_t / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, **SHAPE, "sample": sample},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# Algorithmic work of one launch of each kernel, in units of one causal contraction
# (U) or in bytes for the HBM-bound preparation pass.
KERNEL_WORK = {
    "k_fwd_stats": ("tensor", 1),  # QK^T (the scores, computed once for the extrema)
    "k_fwd_main": ("tensor", 1),   # PV (its QK^T is a recomputation)
    "k_bwd_dq": ("tensor", 2),     # dP = dO V^T, dQ = dS K
    "k_bwd_dkdv": ("tensor", 2),   # dV = P^T dO, dK = dS^T Q (S^T, dP^T are recomputations)
    "k_bwd_fused": ("tensor", 4),  # single pass: dP^T, dV, dK, dQ (S^T is a recomputation)
    # single pass, HBM passes over [B,H,T,d] fp32: the extremum terms read Q, K at the arg-max
    # rows and dQ, write dQ and add to dK (5)
    "k_bwd_ext": ("hbm", 5),
    # per launch, [B,H,T,d] fp32 tensor passes: the forward launch reads V and writes V^T (2),
    # the backward one reads Q, K, dO and O*, writes three transposes and (single pass) zeroes
    # dQ (8); 5 on average
    "k_prep": ("hbm", 5),
}


PROFILE_VARIANTS = {"kint": VARIANT, "softmax": dict(Kint=4, calib=2, tau=8.0, recon=0, ste=0, grad=0),
                    "exp_fp8": dict(Kint=4, calib=4, tau=8.0, recon=0, ste=0, grad=0)}


def profile_steps(args, dev):
    """W + K plain fwd+bwd steps (stream launches, nothing else) of the workload with
    B = --batch and the operator --variant: the program the ncu captures profile."""
    import torch
    from paper_2609_33591_gb300 import kint
    from paper_2609_33591_gb300.inputs import make_qkvdo
    if args.workload == "long":  # the long-context operator (K=16, MinMax, LERP) on --heads heads of T=16384, d=128
        spec = OTHER_CONFIGS["long_context"]
        B, H, T, d = 1, args.heads, spec["shape"][2], spec["shape"][3]
        var = dict(spec["variant"]) if args.variant == "kint" else PROFILE_VARIANTS[args.variant]
        cfg = kint.Config(**var)
        q, k, v, do = (torch.from_numpy(x).to(dev) for x in make_qkvdo(B, H, T, d, seed=spec["seed"]))
    else:
        B, H, T, d = args.batch, SHAPE["H"], SHAPE["T"], SHAPE["d"]
        cfg = kint.Config(**PROFILE_VARIANTS[args.variant])
        q, k, v, do = (torch.from_numpy(x).to(dev) for x in make_qkvdo(B, H, T, d, seed=1))
    for i in range(args.warmup + args.steps):
        O, st = kint.forward(q, k, v, cfg, kint.PREC_TF32)
        kint.backward(q, k, v, O, do, st, cfg, kint.PREC_TF32)
    torch.cuda.synchronize()
    kint.check_status()
    print(json.dumps({"profile_steps": args.warmup + args.steps, "B": B, "H": H, "T": T, "d": d,
                      "variant": args.variant}), flush=True)
    return 0


def run_cuda(args, world, rank, local):
    import torch
    from paper_2609_33591_gb300 import kint
    from paper_2609_33591_gb300.inputs import make_qkvdo

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    kint.load()
    B, H, T, d = SHAPE["B"], SHAPE["H"], SHAPE["T"], SHAPE["d"]
    cfg = kint.Config(**VARIANT)
    prec = kint.PREC_TF32
    if args.profile_steps:
        return profile_steps(args, dev)
    Qh, Kh, Vh, dOh = make_qkvdo(B, H, T, d, seed=1)
    sets = []
    for _ in range(N_INPUT_SETS):
        sets.append(tuple(torch.from_numpy(x).to(dev) for x in (Qh, Kh, Vh, dOh)))
    O = torch.empty_like(sets[0][0])
    grads = tuple(torch.empty_like(sets[0][0]) for _ in range(3))
    st = kint.alloc_rowstats(B, H, T, d, dev, cfg.prob)
    ws_f = kint.workspace(B, H, T, d, prec, 0, dev)
    ws_b = kint.workspace(B, H, T, d, prec, 1, dev)

    def step(i, c=cfg, p=prec):
        q, k, v, do = sets[i % N_INPUT_SETS]
        kint.forward(q, k, v, c, p, O=O, stats=st, ws=ws_f)
        kint.backward(q, k, v, O, do, st, c, p, grads=grads, ws=ws_b)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    def timed(n, fn):
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for i in range(n):
            fn(i)
        e1.record()
        torch.cuda.synchronize()
        barrier()
        return reduce_max(e0.elapsed_time(e1) / n, world, dev)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    kint.check_status()

    # launches per step, counted through the library's launch hook
    per_step = [0]
    kint.kint_set_launch_callback(lambda name, phase, stream: per_step.__setitem__(0, per_step[0] + (phase == 0)))
    step(0)
    kint.kint_set_launch_callback(None)
    torch.cuda.synchronize()

    # The timed steps replay one CUDA graph per input set (the same kernels and launch
    # attributes as the stream calls; the launch overhead of the Python binding stays out)
    graphs = []
    try:
        cs = torch.cuda.Stream()
        cs.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cs):
            for i in range(N_INPUT_SETS):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=cs):
                    step(i)
                graphs.append(g)
        torch.cuda.current_stream().wait_stream(cs)
        for g in graphs:
            g.replay()
        torch.cuda.synchronize()
        kint.check_status()
        launch_mode, run_step = "cuda_graph", (lambda i: graphs[i % N_INPUT_SETS].replay())
    except Exception:  # capture unsupported here: plain stream launches
        graphs = []
        launch_mode, run_step = "stream", step
        torch.cuda.synchronize()

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    ms = timed(args.steps, run_step)
    clocks = sampler.stop()
    kint.check_status()
    launches = [per_step[0] * args.steps]

    # Per-kernel durations: CUDA events on the launching stream around every launch, over a
    # second pass of stream-launched steps (events between launches would otherwise stretch
    # the timed steps by about 25 us each)
    events = {}
    cur_stream = torch.cuda.current_stream()

    def on_launch(name, phase, stream):
        ev = torch.cuda.Event(enable_timing=True)
        ev.record(cur_stream)
        if phase == 0:
            events.setdefault(name, []).append([ev, None])
        else:
            events[name][-1][1] = ev

    n_kt = max(3, min(args.steps, 200))
    kint.kint_set_launch_callback(on_launch)
    timed(n_kt, step)
    kint.kint_set_launch_callback(None)
    kint.check_status()

    per_kernel = {}
    for name, lst in events.items():
        durs = [a.elapsed_time(b) for a, b in lst]
        per_kernel[name] = {"launches": len(durs), "avg_us": 1e3 * sum(durs) / len(durs),
                            "total_ms": sum(durs)}
    flops_step = 6 * unit_flops(B, H, T, d)
    value = job_value(flops_step, world, ms)

    pk = peaks()
    tf32_peak = pk["bf16"] * TF32_PER_BF16
    dom = max(per_kernel, key=lambda n: per_kernel[n]["total_ms"])
    bound, units = KERNEL_WORK[dom]
    avg_s = per_kernel[dom]["avg_us"] * 1e-6
    if bound == "tensor":
        achieved = units * unit_flops(B, H, T, d) / avg_s / 1e12
        traffic = TRAFFIC.get(dom) if TRAFFIC.get("src") == kernel_source_digest() else None
        roof = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": tf32_peak, "unit": "TFLOP/s",
                "frac": achieved / tf32_peak, "traffic": traffic,
                "peak_note": f"TF32 = (1.1 / 2.25 nominal) x {pk['source']} bf16 burst {pk['bf16']} TFLOP/s"}
    else:
        nbytes = units * B * H * T * d * 4
        achieved = nbytes / avg_s / 1e9
        roof = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / pk["hbm_gbs"], "traffic": None}

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "tf32", "data": "synthetic",
            "config": {"workload": WORKLOAD, **SHAPE, **{k: v for k, v in VARIANT.items()}, "prec": "tf32",
                       "launch": launch_mode,
                       "parallelism": f"replicas x{world} (b,h)-sharded, no collective",
                       "l2": f"{N_INPUT_SETS} rotating input sets of {4 * B * H * T * d * 4 >> 20} MiB each; "
                             "per-step traffic (>300 MB) exceeds the 129 MB L2"},
            "tf32_peak_frac": value / world / tf32_peak,
            "roofline": roof, "kernels": per_kernel,
            "kernel_timing": f"CUDA events around each launch on its stream, over a second pass of {n_kt} steps",
            "gpu_launches": launches[0], "clocks": clocks}

    # plain softmax built the same way, and the 3xTF32 mode, on the same inputs
    soft = kint.Config(Kint=4, calib=kint.CALIB_SOFTMAX, tau=8.0, recon=kint.RECON_LERP, ste=0, grad=0)
    n_cmp = max(3, min(args.steps, 200))
    ms_soft = timed(n_cmp, lambda i: step(i, soft, prec))
    line["softmax_comparator"] = {"value": job_value(flops_step, world, ms_soft), "unit": UNIT,
                                  "ms_per_step": ms_soft}
    # the FP8-rounded exponential baseline (E4M3(e^z) forward, e^z backward) on the same inputs
    e8 = kint.Config(Kint=4, calib=kint.CALIB_EXP_FP8, tau=8.0, recon=kint.RECON_LERP, ste=0, grad=0)
    ms_e8 = timed(n_cmp, lambda i: step(i, e8, prec))
    line["exp_fp8_baseline"] = {"value": job_value(flops_step, world, ms_e8), "unit": UNIT, "ms_per_step": ms_e8}
    ws_f3 = kint.workspace(B, H, T, d, kint.PREC_3XTF32, 0, dev)
    ws_b3 = kint.workspace(B, H, T, d, kint.PREC_3XTF32, 1, dev)

    def step3(i):
        q, k, v, do = sets[i % N_INPUT_SETS]
        kint.forward(q, k, v, cfg, kint.PREC_3XTF32, O=O, stats=st, ws=ws_f3)
        kint.backward(q, k, v, O, do, st, cfg, kint.PREC_3XTF32, grads=grads, ws=ws_b3)

    step3(0)
    ms3 = timed(n_cmp, step3)
    line["x3tf32_mode"] = {"value": job_value(flops_step, world, ms3), "unit": UNIT, "ms_per_step": ms3}
    del ws_f3, ws_b3

    # End to end through the public API: every step copies its inputs in from pinned host
    # memory and its results (O, dQ, dK, dV) out.  The copies run on their own streams into
    # and out of two alternating device buffer sets, so step i's compute overlaps step i+1's
    # input copy and step i-1's output copy (host -> device and device -> host at once).
    pin_in = [torch.from_numpy(x).pin_memory() for x in (Qh, Kh, Vh, dOh)]
    pin_out = [torch.empty(B, H, T, d).pin_memory() for _ in range(4)]
    ins = [tuple(torch.empty_like(sets[0][0]) for _ in range(4)) for _ in range(2)]
    outs = [tuple(torch.empty_like(sets[0][0]) for _ in range(4)) for _ in range(2)]
    s_c = torch.cuda.current_stream()
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev = {k: [torch.cuda.Event() for _ in range(2)] for k in ("in", "done", "out")}
    used = set()

    def e2e_step(i):
        b = i % 2
        q, k, v, do = ins[b]
        Ob, dq, dk, dv = outs[b]
        with torch.cuda.stream(s_in):
            if ("done", b) in used:
                s_in.wait_event(ev["done"][b])  # the compute that read this input set finished
            for dst, src in zip(ins[b], pin_in):
                dst.copy_(src, non_blocking=True)
            ev["in"][b].record(s_in)
        s_c.wait_event(ev["in"][b])
        if ("out", b) in used:
            s_c.wait_event(ev["out"][b])  # this output set has been copied out
        kint.forward(q, k, v, cfg, prec, O=Ob, stats=st, ws=ws_f)
        kint.backward(q, k, v, Ob, do, st, cfg, prec, grads=(dq, dk, dv), ws=ws_b)
        ev["done"][b].record(s_c)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev["done"][b])
            for dst, src in zip(pin_out, outs[b]):
                dst.copy_(src, non_blocking=True)
            ev["out"][b].record(s_out)
        used.update((("done", b), ("out", b)))

    def e2e_run(n):
        s_in.wait_stream(s_c)  # the first copy starts inside the timed region
        for i in range(n):
            e2e_step(i)
        s_c.wait_stream(s_out)  # the timed region ends with the last results on the host side

    e2e_run(2)
    n_e2e = max(3, min(args.steps, 100))
    ms_e2e = timed(1, lambda i: e2e_run(n_e2e)) / n_e2e
    # the same copies with no compute, each direction streaming back to back on its own
    # stream: the host link's floor for the end-to-end steps
    def copies_only(n):
        s_in.wait_stream(s_c)
        s_out.wait_stream(s_c)
        for i in range(n):
            with torch.cuda.stream(s_in):
                for dst, src in zip(ins[i % 2], pin_in):
                    dst.copy_(src, non_blocking=True)
            with torch.cuda.stream(s_out):
                for dst, src in zip(pin_out, outs[i % 2]):
                    dst.copy_(src, non_blocking=True)
        s_c.wait_stream(s_in)
        s_c.wait_stream(s_out)

    copies_only(2)
    ms_link = timed(1, lambda i: copies_only(n_e2e)) / n_e2e
    line["e2e"] = {"value": job_value(flops_step, world, ms_e2e), "unit": UNIT,
                   "h2d_bytes_per_step": sum(t.numel() * 4 for t in pin_in),
                   "d2h_bytes_per_step": sum(t.numel() * 4 for t in pin_out), "ms_per_step": ms_e2e,
                   "copies_only_ms_per_step": ms_link, "link_bound_frac": ms_link / ms_e2e}
    kint.check_status()

    # the other configurations' workloads, one at a time (their inputs replace these)
    del sets, O, grads, st, ws_f, ws_b, ins, outs, pin_in, pin_out
    torch.cuda.empty_cache()
    if not args.headline_only:
        line["other_configs"] = {}
        for name, spec in OTHER_CONFIGS.items():
            B2, H2, T2, d2 = spec["shape"]
            Q2, K2, V2, dO2 = (torch.from_numpy(x).to(dev) for x in
                               make_qkvdo(B2, H2, T2, d2, seed=spec["seed"], peaked_frac=spec["peaked"]))
            O2 = torch.empty_like(Q2)
            g2 = tuple(torch.empty_like(Q2) for _ in range(3))
            c2 = kint.Config(**spec["variant"])
            st2 = kint.alloc_rowstats(B2, H2, T2, d2, dev, c2.prob)
            wf2 = kint.workspace(B2, H2, T2, d2, prec, 0, dev)
            wb2 = kint.workspace(B2, H2, T2, d2, prec, 1, dev)

            def step2(i, c=c2):
                kint.forward(Q2, K2, V2, c, prec, O=O2, stats=st2, ws=wf2)
                kint.backward(Q2, K2, V2, O2, dO2, st2, c, prec, grads=g2, ws=wb2)

            for i in range(3):
                step2(i)
            n2 = 5 if T2 <= 4096 else 3
            ms2 = timed(n2, step2)
            f2 = 6 * unit_flops(B2, H2, T2, d2)
            rec = {"workload": spec["workload"], "value": job_value(f2, world, ms2), "unit": UNIT,
                   "ms_per_step": ms2, "steps": n2, "warmup": 3, "tf32_peak_frac": f2 / (ms2 * 1e-3) / 1e12 / tf32_peak,
                   "l2": "inputs larger than the 129 MB L2 (one input set)"}
            if spec["softmax"]:
                for i in range(3):
                    step2(i, soft)
                ms_s = timed(n2, lambda i: step2(i, soft))
                rec["softmax_comparator"] = {"value": job_value(f2, world, ms_s), "unit": UNIT, "ms_per_step": ms_s}
            kint.check_status()
            line["other_configs"][name] = rec
            del Q2, K2, V2, dO2, O2, g2, st2, wf2, wb2
            torch.cuda.empty_cache()
    # a measured TF32 tensor peak on this GPU (cuBLAS), beside the nominal-ratio denominator
    tf32_meas = cublas_tf32_tflops(dev)
    roof["cublas_tf32_measured"] = tf32_meas
    roof["frac_of_cublas_tf32"] = roof["achieved"] / tf32_meas if roof["unit"] == "TFLOP/s" else None
    line["tf32_peak_frac_of_cublas"] = value / world / tf32_meas

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        heads = SHAPE["B"] * SHAPE["H"]
        rate, dt, threads, reps = cpu_oracle_rate(heads, min_seconds=10.0)
        line["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle",
                                "sample": f"the whole workload ({heads} (b,h) heads at T=1024, fwd+bwd) x {reps}, "
                                          f"fp64 oracle, {dt:.1f} s wall on {threads} threads"}
        # the same oracle checks the timed workload's outputs (outside the timed region)
        line["parity"] = bench_parity(Qh, Kh, Vh, dOh)
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["cuda", "reference"], default="cuda")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--headline-only", action="store_true", help="skip the other configurations' lines")
    ap.add_argument("--profile-steps", action="store_true",
                    help="only run warmup + steps plain fwd+bwd steps (B = --batch, operator --variant) for ncu")
    ap.add_argument("--batch", type=int, default=SHAPE["B"])
    ap.add_argument("--variant", choices=sorted(PROFILE_VARIANTS), default="kint")
    ap.add_argument("--workload", choices=["gpt2", "long"], default="gpt2", help="--profile-steps workload")
    ap.add_argument("--heads", type=int, default=8, help="--profile-steps --workload long: heads of T=16384")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    world, rank, local = dist_setup(args.gpus)
    try:
        if args.impl == "reference":
            return run_reference(args, world, rank)
        return run_cuda(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
