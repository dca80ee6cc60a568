#!/usr/bin/env python3
"""Benchmark of the BSR x dense product on one GB300 (or N replicas).

Headline workload: BERT-large's attention projections -- 96 weights (24
layers x Q, K, V, O) of 1024x1024 at 90% block sparsity, in 32x1 and in 16x16
blocks (uniform random block placement, values N(0, 0.02)), fp32 (the paper's
precision), X = 16384x1024 fp32 N(0, 1) shared by every call, bias N(0, 0.02).
One step = one bsr_spmm call per weight and block shape (192 calls, on one
stream, in order), inputs resident in HBM, L2 flushed (a 512 MiB write,
untimed) before every timed step.

Metric: useful GFLOP/s = sum over calls of 2*N*nnz (nnz = stored block
elements) / device time (CUDA events at step boundaries only: consecutive
launches of a step overlap through the library's programmatic launches, and
an event between them would serialise them). Per-step median, p10 and p90,
and the same steps with L2 left warm ("hot_l2"), are reported beside it.
A second pass puts an event pair around every launch to give each kernel's
average duration; the kernel with the largest time share is reported against
its roofline ("roofline"), and the whole step against the sum of its calls'
rooflines ("roofline.step"). The FP32 FMA peak that bounds the SIMT kernels
is measured here, by a probe kernel of packed fp32 multiply-adds on every SM
(burst and sustained). ``e2e`` repeats the step through the C ABI with pinned
host X and Y (the library copies X in and Y out inside every call): on one
stream, and on eight streams as a server would issue independent products.
``cpu_baseline`` times the float-accumulate oracle on one host core and on
every core this process may use. ``workloads`` holds the other benchmark
workloads (one weight at 128 tokens, the block-shape sweep, BERT-base's 48
projections, BERT-large in bf16, the Zipf-row stress weight), each against
its own roofline.

``--workload 1..5`` instead reports one workload (one JSON line per block
shape and dtype), with its step also timed as a captured plan.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
    python bench.py --workload 4 [--steps K] [--dtype bf16] [--shapes 16x16]
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "BSR SpMM GFLOP/s & HBM GB/s vs roofline; BERT attn-projection latency"
WORKLOAD = ("BERT-large attention projections: 96 weights (24 layers x Q,K,V,O) 1024x1024 at 90% block sparsity, "
            "32x1 and 16x16 blocks, fp32; X 16384x1024 fp32 shared by all calls")
HEADLINE_SHAPES = [(32, 1), (16, 16)]
TF32_PER_BF16 = 1.1 / 2.25      # nominal dense tf32 : bf16 tensor rate
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0}
MIN_TIMED_S = 0.5               # at least this much timed work, so the clock sampler sees the region


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer passes (profiling runs)")
    ap.add_argument("--no-extra", action="store_true", help="skip the other workloads (profiling runs)")
    ap.add_argument("--cpu-seconds", type=float, default=16.0)
    ap.add_argument("--workload", type=int, default=0, choices=[0, 1, 2, 3, 4, 5],
                    help="0: the benchmark line; 1-5: a per-workload report (one JSON line per block shape "
                         "and dtype), 1 GPU")
    ap.add_argument("--dtype", default="", help="report only this dtype (f32 or bf16)")
    ap.add_argument("--shapes", default="", help="comma-separated subset of block shapes, e.g. 32x1,16x16")
    ap.add_argument("--weights", type=int, default=0, help="use the first W weights of workloads 3 and 4 only")
    ap.add_argument("--min-seconds", type=float, default=MIN_TIMED_S,
                    help="time at least this long (0: exactly --steps steps; profiling runs)")
    ap.add_argument("--no-probe", action="store_true",
                    help="skip the FP32 peak probe and use the derived peak (profiling runs)")
    return ap.parse_args(argv)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        d["source"] = "measured"
        return d
    d = dict(FALLBACK_PEAKS)
    d["source"] = "fallback"
    return d


def call_bytes(w, N, es):
    """Algorithmic bytes of one call: data + indices + indptr + X + Y + bias, each once."""
    return w.nnz * es + 4 * w.nnzb + 4 * (w.M // w.R + 1) + N * w.K * es + N * w.M * es + 4 * w.M


def pct(xs, q):
    return float(np.percentile(np.asarray(xs, dtype=np.float64), q))


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap,utilization.gpu")

    def __init__(self, index: int):
        self.index = index
        self.samples = []
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.2)   # the sampler is running before the region starts
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == 8:
                self.samples.append(parts)

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}

        def num(s):
            try:
                return float(s)
            except ValueError:
                return None
        busy = [s for s in self.samples if (num(s[7]) or 0) > 0]
        use = busy or self.samples
        sm = [v for v in (num(s[0]) for s in use) if v is not None]
        mx = [v for v in (num(s[1]) for s in self.samples) if v is not None]
        pw = [v for v in (num(s[2]) for s in use) if v is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in use for i in range(4) if s[3 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None, "reasons": reasons, "samples": len(self.samples),
                "samples_under_load": len(busy)}


# ------------------------------------------------------------------ helpers

def dist_setup():
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    """Largest value of x over all ranks (the slowest rank sets the job time)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def source_digest(paths):
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str):
    """DRAM bytes per launch of `kernel` from profiles/dram_traffic.txt, if
    captured on the current kernel sources (else None)."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(p):
        return None
    for line in open(p):
        parts = line.split()
        if len(parts) >= 4 and not line.startswith("#") and parts[0] == kernel:
            src = parts[3].split(",")
            try:
                if source_digest(src[1:]) == src[0]:
                    return float(parts[1])
            except OSError:
                return None
    return None


def dev_array(a, dev):
    import torch
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
    return torch.from_numpy(a).to(dev)


# ------------------------------------------------------------------ FP32 FMA peak

def derived_fp32_peak(dev, pk):
    import torch
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    t = sms * 128 * 2 * float(pk.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
    return {"fma_f32x2_sustained": t, "source": f"derived: {sms} SMs x 128 FP32 lanes x 2 x max clock (not measured)"}


def fp32_peak(dev, stream, sustained_s=1.5):
    """Measured FP32 multiply-add rate (TFLOP/s) of the probe kernel on every
    SM: burst (best of short launches) and sustained (back-to-back launches
    for `sustained_s` seconds, clocks sampled), packed and scalar FMA."""
    import torch
    from paper_2106_08846_gb300 import _build
    lib = ctypes.CDLL(_build.build_probe())
    lib.bsr_probe_fma.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int64, ctypes.c_int,
                                  ctypes.c_void_p]
    lib.bsr_probe_fma_count.restype = ctypes.c_int64
    lib.bsr_probe_fma_count.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64]
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    blocks, threads = sms * 8, 256
    out = torch.empty(blocks * threads, dtype=torch.float32, device=dev)
    sp = ctypes.c_void_p(stream.cuda_stream)

    def run(iters, packed, reps=1):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            if lib.bsr_probe_fma(ctypes.c_void_p(out.data_ptr()), blocks, threads, iters, packed, sp) != 0:
                raise RuntimeError("FP32 probe launch failed")
        e1.record(stream)
        torch.cuda.synchronize()
        return 2.0 * reps * lib.bsr_probe_fma_count(blocks, threads, iters) / (e0.elapsed_time(e1) * 1e-3) / 1e12

    res = {}
    it = 2000
    run(it, 1)
    t = 2.0 * lib.bsr_probe_fma_count(blocks, threads, it) / (run(it, 1) * 1e12)
    it = max(1000, int(it * 0.02 / t))   # about 20 ms per launch
    for packed, key in ((1, "fma_f32x2"), (0, "fma_f32")):
        res[key + "_burst"] = max(run(it, packed) for _ in range(5))
    reps = max(1, int(sustained_s / 0.02))
    with ClockSampler(dev.index or 0) as clk:
        res["fma_f32x2_sustained"] = run(it, 1, reps)
    res["clocks"] = clk.summary()
    res["launch"] = f"{blocks} CTAs x {threads} threads, {it} iterations of 16 multiply-adds per thread"
    return res


# ------------------------------------------------------------------ CPU oracle

def cpu_threads():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def time_cpu(bsrs, weights, X, threads, seconds):
    """The float-accumulate oracle over (weight, BSR) pairs on X's tokens, on
    `threads` cores, repeated until `seconds` pass (at least once).
    Returns (GFLOP/s, repetitions)."""
    import oracle
    flops, elapsed, reps = 0, 0.0, 0
    while elapsed < seconds or reps == 0:
        for w, b in zip(weights, bsrs):
            t0 = time.perf_counter()
            oracle.bsr_spmm_f32acc(*b, X, w.bias, w.M, threads=threads)
            elapsed += time.perf_counter() - t0
            flops += 2 * X.shape[0] * w.nnz
        reps += 1
    return flops / elapsed / 1e9, reps


def headline_weights(dtype="f32", only=None):
    import synth
    ws = []
    for shape in HEADLINE_SHAPES:
        ws += synth.config(4, dtype=dtype, shape=shape, only=only).weights
    return ws


def cpu_baseline(args, weights_by_shape, X_np):
    """One representative weight per block shape (the first, layer 0's Q),
    on a token sample sized for about cpu_seconds of CPU work in all."""
    import oracle
    oracle.build()
    ws = [w for w in weights_by_shape]
    bsrs = [oracle.bsr_from_dense(w.W, w.R, w.C) for w in ws]
    ncores = min(cpu_threads(), oracle.max_threads())
    # calibrate the sample: tokens for about a quarter of the budget on one core
    probe = X_np[:8]
    g1, _ = time_cpu(bsrs, ws, probe, 1, 0.0)
    flops_per_token = sum(2 * w.nnz for w in ws)
    tokens = int(np.clip(g1 * 1e9 * (args.cpu_seconds / 4) / flops_per_token, 8, X_np.shape[0]))
    Xs = X_np[:tokens]
    single, r1 = time_cpu(bsrs, ws, Xs, 1, args.cpu_seconds / 2)
    multi, rn = time_cpu(bsrs, ws, Xs, ncores, args.cpu_seconds / 2)
    shapes = ",".join(f"{w.R}x{w.C}" for w in ws)
    return {"value": multi, "unit": "GFLOP/s", "cores": ncores, "kind": "oracle",
            "sample": (f"float-accumulate oracle (ref_bsr_spmm_f32acc), OpenMP over block rows; one 1024x1024 "
                       f"weight per block shape ({shapes}) x the first {tokens} of 16384 tokens, {rn} passes; the "
                       f"96-weight step scales by weight count"),
            "single_core": {"value": single, "cores": 1, "passes": r1}}


def run_reference(args, world, rank):
    """The oracle as it stands, on the host cores: each step the float-
    accumulate oracle over every weight of the headline workload on a
    bounded token sample, block rows shared among all cores."""
    if rank != 0:
        return
    import oracle
    import synth
    oracle.build()
    ws = headline_weights()
    N_full = synth.config(4, only=[0]).N
    tokens = 8
    X = synth.config(4, only=[0]).make_X(N=tokens)
    bsrs = [oracle.bsr_from_dense(w.W, w.R, w.C) for w in ws]
    ncores = min(cpu_threads(), oracle.max_threads())

    def step():
        t0 = time.perf_counter()
        for w, b in zip(ws, bsrs):
            oracle.bsr_spmm_f32acc(*b, X, w.bias, w.M, threads=ncores)
        return time.perf_counter() - t0

    for _ in range(args.warmup):
        step()
    times = [step() for _ in range(args.steps)]
    flops = sum(2 * tokens * w.nnz for w in ws)
    total = sum(times)
    value = flops * args.steps / total / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": WORKLOAD, "N": N_full, "M": 1024, "K": 1024, "sparsity": 90,
                   "shapes": [f"{r}x{c}" for r, c in HEADLINE_SHAPES], "weights_per_shape": 96},
        "cpu_baseline": {"value": value, "unit": "GFLOP/s", "cores": ncores, "kind": "oracle",
                         "sample": f"every weight of the step (2 x 96) on the first {tokens} of {N_full} tokens "
                                   f"per step; float-accumulate oracle, OpenMP over block rows"},
        "e2e": {"value": value, "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU measurement

class Product:
    """The handles and buffers of one workload on the device."""

    def __init__(self, bsr, weights, X, N, dev):
        import torch
        self.weights, self.X, self.N = weights, X, N
        self.es = 2 if X.dtype == torch.bfloat16 else 4
        self.handles, self.biases = [], []
        for w in weights:
            arrays = bsr.bsr_from_dense(dev_array(w.W, dev), w.R, w.C, 0.0)
            h = bsr.bsr_create(*arrays, w.R, w.C, w.M, w.K)
            h.reserve(N)
            self.handles.append(h)
            self.biases.append(torch.from_numpy(w.bias).to(dev))
        self.Y = torch.empty((N, weights[0].M), dtype=X.dtype, device=dev)   # every weight here is M x K
        self.scheds = [h.schedule() for h in self.handles]
        self.flops = [2 * N * w.nnz for w in weights]
        self.nbytes = [call_bytes(w, N, self.es) for w in weights]
        self.bsr = bsr

    def step(self, stream):
        for h, b in zip(self.handles, self.biases):
            self.bsr.bsr_spmm(h, self.X, b, self.Y, self.N, stream)

    def launches(self):
        return sum(s["launches_per_call"] for s in self.scheds)

    def check(self):
        for h in self.handles:
            if h.check_device_status() != 0:
                raise RuntimeError("device status error")

    def destroy(self):
        for h in self.handles:
            h.destroy()


def kernel_key(sc, w):
    return f"{sc['variant']}_{w.R}x{w.C}_{'bf16' if w.dtype == 'bf16' else 'f32'}"


def pipe_peak(sc, dtype, pk, fp32_tflops):
    """(peak FLOP/s, description) of the pipe that bounds this kernel's arithmetic."""
    if sc["variant"] == "tcgen05":
        bf16 = float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"])) * 1e12
        if dtype == "bf16":
            return bf16, f"bf16 tensor, sustained ({pk['source']})"
        return bf16 * TF32_PER_BF16 / 3.0, (f"3xTF32: tf32 tensor (bf16 sustained x {TF32_PER_BF16:.3f}, "
                                             f"{pk['source']}) / 3 products")
    return fp32_tflops * 1e12, "FP32 FMA, measured sustained (packed fma.rn.f32x2 probe)"


def timed_steps(prod_steps, K, stream, flush, hold_s=0.0):
    """K steps, each bracketed by CUDA events (L2 flushed before each when
    `flush` is given). The stream is first held for `hold_s` so that the
    host enqueues ahead of the device. Returns per-step milliseconds."""
    import torch
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    if hold_s > 0:
        torch.cuda._sleep(int(hold_s * 2.0e9))
    for k in range(K):
        if flush is not None:
            flush.zero_()
        ev[k][0].record(stream)
        prod_steps()
        ev[k][1].record(stream)
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in ev]


def per_call_ms(prod, K, stream, flush):
    """Average duration of every call, from an event pair around each launch."""
    import torch
    n = len(prod.handles)
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
          for _ in range(K)]
    for k in range(K):
        flush.zero_()
        for i, (h, b) in enumerate(zip(prod.handles, prod.biases)):
            ev[k][i][0].record(stream)
            prod.bsr.bsr_spmm(h, prod.X, b, prod.Y, prod.N, stream)
            ev[k][i][1].record(stream)
    torch.cuda.synchronize()
    return [statistics.fmean(ev[k][i][0].elapsed_time(ev[k][i][1]) for k in range(K)) for i in range(n)]


def enqueue_seconds(prod, stream):
    import torch
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    prod.step(stream)
    s = time.perf_counter() - t0
    torch.cuda.synchronize()
    return s


def measure(prod, K_req, warmup, stream, flush, pk, fp32_tflops, hbm, world=1, clocks_index=None,
            min_s=MIN_TIMED_S):
    """Step times (flushed and hot L2), per-kernel roofline and the step roofline."""
    import torch
    for _ in range(max(warmup, 3)):
        flush.zero_()
        prod.step(stream)
    torch.cuda.synchronize()
    one = timed_steps(lambda: prod.step(stream), 1, stream, flush)[0] * 1e-3
    K = max(K_req, int(math.ceil(min_s / max(one, 1e-6))))
    enq = enqueue_seconds(prod, stream)
    hold = min(enq * K * 1.5 + 0.01, 2.0)
    barrier(world)
    sampler = ClockSampler(clocks_index) if clocks_index is not None else None
    if sampler:
        sampler.__enter__()
    try:
        flushed = timed_steps(lambda: prod.step(stream), K, stream, flush, hold)
    finally:
        if sampler:
            sampler.__exit__(None, None, None)
    barrier(world)
    hot = timed_steps(lambda: prod.step(stream), K, stream, None, hold)
    calls = per_call_ms(prod, max(1, min(K, 20)), stream, flush)
    prod.check()

    # roofline of every call: the slower of its FLOPs at its pipe's peak and its bytes at HBM
    roof_s, kinds = [], {}
    for i, (w, sc) in enumerate(zip(prod.weights, prod.scheds)):
        peak, desc = pipe_peak(sc, w.dtype, pk, fp32_tflops)
        roof_s.append(max(prod.flops[i] / peak, prod.nbytes[i] / hbm))
        key = kernel_key(sc, w)
        d = kinds.setdefault(key, {"ms": 0.0, "calls": 0, "flops": 0, "bytes": 0, "roof_s": 0.0, "peak": peak,
                                   "peak_desc": desc, "sc": sc, "w": w})
        d["ms"] += calls[i]
        d["calls"] += 1
        d["flops"] += prod.flops[i]
        d["bytes"] += prod.nbytes[i]
        d["roof_s"] += roof_s[-1]
    total_ms = sum(flushed)
    step_ms = statistics.median(flushed)
    res = {
        "K": K, "total_ms": total_ms, "step_ms": step_ms,
        "p10_ms": pct(flushed, 10), "p90_ms": pct(flushed, 90), "mean_ms": total_ms / K,
        "hot_ms": statistics.median(hot), "hot_p10_ms": pct(hot, 10), "hot_p90_ms": pct(hot, 90),
        "flops": sum(prod.flops), "bytes": sum(prod.nbytes), "roof_ms": sum(roof_s) * 1e3,
        "clocks": sampler.summary() if sampler else None, "kinds": kinds, "calls_ms": calls,
    }
    return res


def kernel_roofline(d, hbm):
    """The roofline object of one kernel kind (average over its calls)."""
    t = d["ms"] / d["calls"] * 1e-3
    flops, nbytes = d["flops"] / d["calls"], d["bytes"] / d["calls"]
    by_bytes = nbytes / hbm >= flops / d["peak"]
    sc, w = d["sc"], d["w"]
    if by_bytes:
        r = {"bound": "hbm", "achieved": nbytes / t / 1e9, "peak": hbm / 1e9, "unit": "GB/s",
             "peak_source": "HBM copy bandwidth, MEASURED_PEAKS.json"}
    else:
        r = {"bound": "alu" if sc["variant"] != "tcgen05" else "tensor", "achieved": flops / t / 1e12,
             "peak": d["peak"] / 1e12, "unit": "TFLOP/s", "peak_source": d["peak_desc"]}
    r["frac"] = r["achieved"] / r["peak"]
    r["traffic"] = profiled_traffic(kernel_key(sc, w) + f"_{w.M}x{w.K}")
    r["kernel"] = (f"{sc['variant']} {w.R}x{w.C} {w.dtype}" +
                   (f" (exec {sc['exec_R']}x{sc['exec_C']})" if (sc['exec_R'], sc['exec_C']) != (w.R, w.C) else ""))
    r["us_per_launch"] = t * 1e6
    r["flops_per_launch"] = flops
    r["bytes_per_launch"] = nbytes
    r["hbm_frac"] = nbytes / t / hbm
    r["roofline_frac"] = max(flops / d["peak"], nbytes / hbm) / t
    return r


def run_e2e(bsr, prod, X_np, K, world, n_streams):
    """The step through the C ABI with pinned host X and Y: every call copies
    X in and Y out inside the call, so the copies are timed. Calls go round-
    robin to `n_streams` streams (one: a plain sequential caller; several: a
    server issuing independent products, whose copies then overlap other
    calls' kernels). Returns (GFLOP/s, h2d bytes, d2h bytes) per step."""
    import torch
    Xh = torch.from_numpy(X_np).pin_memory()   # fp32 (the headline workload)
    streams = [torch.cuda.Stream() for _ in range(n_streams)]
    Yh = [torch.empty((prod.N, prod.weights[0].M), dtype=prod.Y.dtype).pin_memory() for _ in streams]
    main = torch.cuda.current_stream()

    def e2e_step():
        for i, (h, b) in enumerate(zip(prod.handles, prod.biases)):
            bsr.bsr_spmm(h, Xh, b, Yh[i % n_streams], prod.N, streams[i % n_streams])

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(main)
    for st in streams:
        st.wait_event(e0)
    for _ in range(K):
        e2e_step()
    for st in streams:   # the region ends when every stream's last call has finished
        done = torch.cuda.Event()
        done.record(st)
        main.wait_event(done)
    e1.record(main)
    torch.cuda.synchronize()
    prod.check()
    ms = max_over_ranks(e0.elapsed_time(e1), world)
    value = world * sum(prod.flops) * K / (ms * 1e-3) / 1e9
    h2d = len(prod.handles) * prod.N * prod.weights[0].K * prod.es
    d2h = len(prod.handles) * prod.N * prod.weights[0].M * prod.es
    return value, h2d, d2h, ms / K


EXTRA = [
    # (key, workload, dtype, shape)
    ("1_bert_base_single_32x1_f32", 1, None, None),
    ("2_sweep_f32", 2, None, None),
    ("3_bert_base_48_32x1_f32", 3, None, None),
    ("4_bert_large_32x1_bf16", 4, "bf16", (32, 1)),
    ("4_bert_large_16x16_bf16", 4, "bf16", (16, 16)),
    ("5_zipf_32x1_bf16", 5, None, (32, 1)),
    ("5_zipf_16x16_bf16", 5, None, (16, 16)),
]


def workload_entry(res, prod, hbm, fp32_tflops):
    kinds = {k: kernel_roofline(d, hbm) for k, d in res["kinds"].items()}
    w0 = prod.weights[0]
    return {
        "weights": len(prod.weights), "N": prod.N, "M": w0.M, "K": w0.K, "dtype": w0.dtype,
        "shapes": sorted({f"{w.R}x{w.C}" for w in prod.weights}),
        "us_per_step": res["step_ms"] * 1e3, "p10_us": res["p10_ms"] * 1e3, "p90_us": res["p90_ms"] * 1e3,
        "hot_l2_us": res["hot_ms"] * 1e3, "steps": res["K"],
        "gflops": res["flops"] / (res["step_ms"] * 1e-3) / 1e9, "gbs": res["bytes"] / (res["step_ms"] * 1e-3) / 1e9,
        "roofline": {"us_per_step": res["roof_ms"] * 1e3, "frac": res["roof_ms"] / res["step_ms"]},
        "kernels": {k: {"us": round(v["us_per_launch"], 2), "frac": round(v["frac"], 4), "bound": v["bound"],
                        "kernel": v["kernel"]} for k, v in kinds.items()},
        "l2": "flushed before every step (hot_l2: not flushed)",
    }


def run_ours(args, world, rank, local):
    import torch

    import synth
    import paper_2106_08846_gb300 as bsr
    from paper_2106_08846_gb300 import _build

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0:
        _build.build()
    barrier(world)
    bsr.load()
    stream = torch.cuda.current_stream()
    pk = peaks()
    hbm = float(pk["hbm_gbs"]) * 1e9
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    fp32 = derived_fp32_peak(dev, pk) if args.no_probe else fp32_peak(dev, stream)
    fp32_tflops = fp32["fma_f32x2_sustained"]

    only = list(range(args.weights)) if args.weights else None
    weights = headline_weights(only=only)
    if args.shapes:
        keep = set(args.shapes.split(","))
        weights = [w for w in weights if f"{w.R}x{w.C}" in keep]
    wl0 = synth.config(4, only=[0])
    X_np = wl0.make_X()
    N = wl0.N
    X = torch.from_numpy(X_np).to(dev)
    prod = Product(bsr, weights, X, N, dev)

    res = measure(prod, args.steps, args.warmup, stream, flush, pk, fp32_tflops, hbm, world, local,
                  args.min_seconds)
    K = res["K"]
    total_ms = max_over_ranks(res["total_ms"], world)
    value = world * res["flops"] * K / (total_ms * 1e-3) / 1e9
    gbs = world * res["bytes"] * K / (total_ms * 1e-3) / 1e9

    # the dominant kernel kind against its roofline
    kinds = {k: kernel_roofline(d, hbm) for k, d in res["kinds"].items()}
    dom = max(res["kinds"], key=lambda k: res["kinds"][k]["ms"])
    roofline = dict(kinds[dom])
    roofline["time_share"] = res["kinds"][dom]["ms"] / sum(d["ms"] for d in res["kinds"].values())
    roofline["step"] = {"roofline_ms": res["roof_ms"], "measured_ms": res["step_ms"],
                        "frac": res["roof_ms"] / res["step_ms"],
                        "definition": "sum over the step's calls of max(FLOPs / pipe peak, algorithmic bytes / HBM)"}
    roofline["kernels"] = kinds

    e2e = None
    if not args.no_e2e:
        v1, h2d, d2h, ms1 = run_e2e(bsr, prod, X_np, max(2, min(K, 5)), world, 1)
        v8, _, _, ms8 = run_e2e(bsr, prod, X_np, max(2, min(K, 5)), world, 8)
        e2e = {"value": v1, "unit": "GFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": ms1,
               "how": "every call through bsr_spmm with pinned host X and Y (copied in and out inside the call), "
                      "one stream",
               "multi_stream": {"value": v8, "streams": 8, "ms_per_step": ms8,
                                "how": "the same calls spread round-robin over 8 streams (a server issuing "
                                       "independent products: copies overlap other calls' kernels)"}}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        reps = []
        for shape in HEADLINE_SHAPES:
            reps += [w for w in weights if (w.R, w.C) == shape][:1]
        cpu = cpu_baseline(args, reps, X_np)

    extra = {}
    if rank == 0 and world == 1 and not args.no_extra:
        for key, k, dt, shape in EXTRA:
            if k == 4:
                ws = synth.config(4, dtype=dt, shape=shape, only=only).weights
                Xe = X.to(torch.bfloat16)
                Ne = N
            else:
                wl = synth.config(k, dtype=dt, shape=shape)
                ws, Ne = wl.weights, wl.N
                Xe = dev_array(wl.make_X(), dev)
            pe = Product(bsr, ws, Xe, Ne, dev)
            r = measure(pe, args.steps, args.warmup, stream, flush, pk, fp32_tflops, hbm, 1, None, args.min_seconds)
            extra[key] = workload_entry(r, pe, hbm, fp32_tflops)
            pe.destroy()
            del Xe

    if rank == 0:
        clocks = res["clocks"] or {}
        line = {
            "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": world, "steps": K,
            "steps_requested": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": total_ms / K,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": WORKLOAD, "N": N, "M": 1024, "K": 1024, "sparsity": 90,
                       "shapes": sorted({f"{w.R}x{w.C}" for w in weights}),
                       "weights_per_shape": len(weights) // max(1, len({(w.R, w.C) for w in weights})),
                       "calls_per_step": len(weights),
                       "l2": "flushed before every timed step (512 MiB write, untimed); X (67 MB) is shared by the "
                             "step's calls and stays in L2 within a step",
                       "parallelism": f"replicas x{world}" if world > 1 else "1 GPU"},
            "step_ms": {"median": res["step_ms"], "p10": res["p10_ms"], "p90": res["p90_ms"]},
            "hot_l2": {"median_ms": res["hot_ms"], "p10_ms": res["hot_p10_ms"], "p90_ms": res["hot_p90_ms"],
                       "gflops": res["flops"] / (res["hot_ms"] * 1e-3) / 1e9},
            "gbs": gbs, "gpu_launches": prod.launches() * K,
            "clocks": dict(clocks, ms_x_mhz=(total_ms / K) * clocks["sm_mhz"] if clocks.get("sm_mhz") else None),
            "fp32_peak": fp32,
            "e2e": e2e,
            "roofline": roofline,
            "cpu_baseline": cpu,
            "workloads": extra,
        }
        print(json.dumps(line), flush=True)
    prod.destroy()


# ------------------------------------------------------------------ per-workload report

REPORT_VARIANTS = {
    1: [(None, None)],
    2: [(None, None)],
    3: [(None, None)],
    4: [("f32", (32, 1)), ("f32", (16, 16)), ("bf16", (32, 1)), ("bf16", (16, 16))],
    5: [(None, (32, 1)), (None, (16, 16))],
}


def run_report(args):
    """One JSON line per block shape and dtype of one workload; workloads of
    several weights are also timed as a captured plan."""
    import torch

    import synth
    import paper_2106_08846_gb300 as bsr
    from paper_2106_08846_gb300 import _build

    _build.build()
    bsr.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    pk = peaks()
    hbm = float(pk["hbm_gbs"]) * 1e9
    stream = torch.cuda.current_stream()
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    fp32 = derived_fp32_peak(dev, pk) if args.no_probe else fp32_peak(dev, stream, sustained_s=0.5)
    fp32_tflops = fp32["fma_f32x2_sustained"]
    for dt, shape in REPORT_VARIANTS[args.workload]:
        if args.dtype and dt is not None and dt != args.dtype:
            continue
        if args.shapes and shape is not None and f"{shape[0]}x{shape[1]}" not in args.shapes.split(","):
            continue
        only = list(range(args.weights)) if args.weights and args.workload in (3, 4) else None
        wl = synth.config(args.workload, dtype=dt, shape=shape, only=only)
        if args.shapes and args.workload == 2:
            wl.weights = [w for w in wl.weights if f"{w.R}x{w.C}" in args.shapes.split(",")]
        X = dev_array(wl.make_X(), dev)
        prod = Product(bsr, wl.weights, X, wl.N, dev)
        res = measure(prod, args.steps, args.warmup, stream, flush, pk, fp32_tflops, hbm, 1, 0, args.min_seconds)
        line = {"workload": args.workload, "name": wl.name}
        line.update(workload_entry(res, prod, hbm, fp32_tflops))
        line["clocks"] = res["clocks"]
        line["fp32_peak_tflops"] = fp32_tflops
        if len(prod.handles) > 1:
            # the same step as one captured plan: the call sequence kept, and
            # (the products being independent) regrouped and fused
            for key, indep in (("plan_sequence", False), ("plan_fused", True)):
                Ys = [torch.empty_like(prod.Y) for _ in prod.handles] if indep else [prod.Y] * len(prod.handles)
                plan = bsr.bsr_plan_create(prod.handles, [X] * len(prod.handles), prod.biases, Ys, independent=indep)
                times = timed_steps(lambda: plan.launch(stream), res["K"], stream, flush)
                order, call, n_kernels = plan.order()
                line[key] = {"us_per_step": statistics.median(times) * 1e3, "library_calls": len(set(call)),
                             "kernels": n_kernels}
                plan.destroy()
        print(json.dumps(line), flush=True)
        prod.destroy()


def main():
    args = parse()
    if args.workload:
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable": "the per-workload report times the GPU path only"}))
            return
        run_report(args)
        return
    world, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
