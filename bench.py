#!/usr/bin/env python3
"""Benchmark of the BSR x dense product on one GB300 (or N replicas).

Workload: the block-shape sweep -- a 768x768 fp32 weight at 80% block
sparsity for each of the block shapes 1x1, 4x4, 8x1, 16x1, 32x1, 1x32, 16x16,
32x32 (uniform random block placement, values N(0, 0.02)), X = 1024x768 fp32
N(0, 1), bias N(0, 0.02). One step = one bsr_spmm call per shape (8 calls).

Metric: useful GFLOP/s = sum over calls of 2*N*nnz (nnz = stored block
elements) / device time, inputs resident in HBM, L2 flushed (a 512 MiB write)
before every timed step and not timed. The timed steps carry CUDA events
only at step boundaries: consecutive launches of a step overlap (each kernel
starts its prologue while the previous one finishes, see the library's
programmatic launches), and an event between them would serialise them. A
second pass over the same steps, inside the same clock-sampled region, puts
an event pair around every launch to give each kernel's average duration
(per_shape); the kernel with the largest share is reported against its
roofline. ``e2e`` repeats the step through the C ABI
with pinned host X and Y (the library copies in and out on the call's stream;
each weight's calls on a stream of their own).
``cpu_baseline`` times the CPU oracle on the host cores.

``--workload 1|3|4|5`` instead reports another benchmark workload (one JSON
line per block shape and dtype): its step as the workload defines it (one
bsr_spmm call per weight, in order, on one stream; L2 flushed before every
step), GFLOP/s and GB/s, and the fraction of the workload's roofline, the
slower of its FLOPs at the arithmetic peak (fp32: the FP32 FMA peak; bf16:
the measured bf16 tensor peak) and its bytes (block values, indices, indptr,
X, Y, bias, each once per call) at the measured HBM bandwidth.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
    python bench.py --workload 4 [--steps K]
"""
from __future__ import annotations

import argparse
import hashlib
import json
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
WORKLOAD = "block-shape sweep: 768x768 fp32 weight at 80% block sparsity, 8 block shapes, X 1024x768 fp32"
FP32_LANES_PER_SM = 128        # FP32 FMA lanes per SM (4 SM sub-partitions x 32)
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "sm_max_mhz": 2070.0}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)   # about 0.4 s timed: several clock samples
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer pass (profiling runs)")
    ap.add_argument("--shapes", default="", help="comma-separated subset of block shapes, e.g. 1x1,32x1 (profiling runs)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--workload", type=int, default=2, choices=[1, 2, 3, 4, 5],
                    help="2: the block-shape sweep (the benchmark line); 1, 3, 4, 5: a per-workload report "
                         "(one JSON line per block shape and dtype, device time against the roofline), 1 GPU")
    ap.add_argument("--dtype", default="", help="report only this dtype (f32 or bf16; profiling runs)")
    ap.add_argument("--weights", type=int, default=0, help="report on the first W weights only (profiling runs)")
    return ap.parse_args()


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


def workload_bytes(w, N, es=4):
    """Algorithmic bytes of one call: data + indices + indptr + X + Y + bias, each once."""
    return (w.nnz * es + 4 * w.nnzb + 4 * (w.M // w.R + 1) + N * w.K * es + N * w.M * es + 4 * w.M)


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

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
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == 7:
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
        sm = [float(s[0]) for s in self.samples if s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in self.samples if s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in self.samples for i in range(4) if s[3 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.samples)}


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
    """dram bytes per launch from profiles/dram_traffic.txt, if taken on the current source."""
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


# ------------------------------------------------------------------ CPU oracle

def time_oracle(wl, bsrs, X, seconds: float, tokens=None):
    """Runs the oracle over the workload (optionally a token subset) until `seconds` pass."""
    import oracle
    rows = None if tokens is None else np.arange(tokens)
    n = wl.N if tokens is None else tokens
    flops, elapsed, reps = 0, 0.0, 0
    while elapsed < seconds or reps == 0:
        for w, b in zip(wl.weights, bsrs):
            t0 = time.perf_counter()
            oracle.bsr_spmm(*b, X, w.bias, w.M, rows=rows)
            elapsed += time.perf_counter() - t0
            flops += 2 * n * w.nnz
        reps += 1
        if reps >= 50:
            break
    return flops, elapsed, reps


def run_reference(args, world, rank):
    if rank != 0:
        return
    import oracle
    import synth
    oracle.build()
    wl = synth.config(2)
    X = wl.make_X()
    bsrs = [oracle.bsr_from_dense(w.W, w.R, w.C) for w in wl.weights]
    tokens = 64                      # bounded sample of the step: 64 of 1024 tokens per shape
    for _ in range(args.warmup):
        time_oracle(wl, bsrs, X, 0.0, tokens)
    times, flops = [], 0
    for _ in range(args.steps):
        f, t, _ = time_oracle(wl, bsrs, X, 0.0, tokens)
        times.append(t)
        flops += f
    total = sum(times)
    value = flops / total / 1e9
    sample = f"{tokens} of {wl.N} tokens per shape per step, all 8 shapes, single thread"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": WORKLOAD, "N": wl.N, "M": 768, "K": 768, "sparsity": 80,
                                        "shapes": [f"{w.R}x{w.C}" for w in wl.weights]},
        "cpu_baseline": {"value": value, "unit": "GFLOP/s", "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU arm

def run_e2e(bsr, handles, biases, wl, X_np, N, K, stream, world, flops_step):
    """The step through the C ABI with pinned host X and Y: each call copies X
    in and Y out (inside the call), so the copies are timed. Each weight's
    calls run on a stream of their own, as a server would issue independent
    layers' products: one call's copies then overlap another call's kernel
    (the host link, about 175 GB/s each way here, carries 50 MB per step)."""
    import torch
    Xh = torch.from_numpy(X_np).pin_memory()
    Yh = [torch.empty((N, w.M), dtype=torch.float32).pin_memory() for w in wl.weights]
    streams = [torch.cuda.Stream() for _ in handles]
    for h, Y, st in zip(handles, Yh, streams):
        bsr.bsr_spmm(h, Xh, None, Y, N, st)       # sizes the staging buffers
    torch.cuda.synchronize()

    def e2e_step():
        for h, b, Y, st in zip(handles, biases, Yh, streams):
            bsr.bsr_spmm(h, Xh, b, Y, N, st)

    for _ in range(3):
        e2e_step()
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for st in streams:
        st.wait_event(e0)
    for _ in range(K):
        e2e_step()
    for st in streams:   # the timed region ends when every stream's last call has finished
        done = torch.cuda.Event()
        done.record(st)
        stream.wait_event(done)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world)
    value = world * flops_step * K / (e2e_ms * 1e-3) / 1e9
    h2d = sum(N * w.K * 4 for w in wl.weights)
    d2h = sum(N * w.M * 4 for w in wl.weights)
    return value, h2d, d2h


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

    wl = synth.config(2)
    if args.shapes:
        keep = set(args.shapes.split(","))
        wl.weights = [w for w in wl.weights if f"{w.R}x{w.C}" in keep]
    N = wl.N
    X_np = wl.make_X()
    X = torch.from_numpy(X_np).to(dev)
    handles, Ys, biases, flops, nbytes = [], [], [], [], []
    for w in wl.weights:
        Wd = torch.from_numpy(w.W).to(dev)
        arrays = bsr.bsr_from_dense(Wd, w.R, w.C, 0.0)
        h = bsr.bsr_create(*arrays, w.R, w.C, w.M, w.K)
        h.reserve(N)
        handles.append(h)
        Ys.append(torch.empty((N, w.M), dtype=torch.float32, device=dev))
        biases.append(torch.from_numpy(w.bias).to(dev))
        flops.append(2 * N * w.nnz)
        nbytes.append(workload_bytes(w, N))
    scheds = [h.schedule() for h in handles]
    launches_per_step = sum(s["launches_per_call"] for s in scheds)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        for h, b, Y in zip(handles, biases, Ys):
            bsr.bsr_spmm(h, X, b, Y, N, stream)

    for _ in range(max(args.warmup, 3)):
        flush.zero_()
        step()
    torch.cuda.synchronize()

    # time the CPU enqueue of one step so the GPU can be held back long enough
    t0 = time.perf_counter()
    step()
    torch.cuda.synchronize()
    enqueue_s = time.perf_counter() - t0
    K = args.steps
    nshape = len(handles)
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nshape)]
          for _ in range(K)]
    st = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    clock_mhz = float(peaks().get("sm_max_mhz", 2070.0))

    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clocks:
        # hold the stream while the host enqueues every timed launch, so that
        # the events time back-to-back device execution, not host launch gaps
        torch.cuda._sleep(int((enqueue_s * K * 2.0 + 0.05) * clock_mhz * 1e6))
        # the timed steps: events only at step boundaries, so that nothing
        # sits between the launches of a step (an event record there would
        # stop a kernel from starting while the previous one finishes)
        for k in range(K):
            flush.zero_()
            st[k][0].record(stream)
            step()
            st[k][1].record(stream)
        torch.cuda.synchronize()
        # per-kernel durations: the same steps again with an event pair
        # around every launch (for per_shape and the roofline)
        torch.cuda._sleep(int((enqueue_s * K * 2.0 + 0.05) * clock_mhz * 1e6))
        for k in range(K):
            flush.zero_()
            for i, (h, b, Y) in enumerate(zip(handles, biases, Ys)):
                ev[k][i][0].record(stream)
                bsr.bsr_spmm(h, X, b, Y, N, stream)
                ev[k][i][1].record(stream)
        torch.cuda.synchronize()
    barrier(world)
    step_ms = [a.elapsed_time(b) for a, b in st]
    total_ms = max_over_ranks(sum(step_ms), world)
    kern_ms = [statistics.fmean(ev[k][i][0].elapsed_time(ev[k][i][1]) for k in range(K)) for i in range(nshape)]
    flops_step = sum(flops)
    value = world * flops_step * K / (total_ms * 1e-3) / 1e9
    gbs = world * sum(nbytes) * K / (total_ms * 1e-3) / 1e9

    # ---- e2e: pinned host X and Y through the C ABI (copies inside the call)
    e2e_value = None
    if not args.no_e2e:
        e2e_value, h2d, d2h = run_e2e(bsr, handles, biases, wl, X_np, N, K, stream, world, flops_step)
    else:
        h2d = d2h = 0

    # ---- dominant kernel vs its roofline
    shares = [kern_ms[i] for i in range(nshape)]
    dom = int(np.argmax(shares))
    w = wl.weights[dom]
    pk = peaks()
    props = torch.cuda.get_device_properties(dev)
    alu_peak_tflops = props.multi_processor_count * FP32_LANES_PER_SM * 2 * float(pk.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
    kern_name = f"bsr_spmm_{w.R}x{w.C}_f32"
    variant = scheds[dom]["variant"]
    achieved = flops[dom] / (kern_ms[dom] * 1e-3) / 1e12
    roofline = {
        "bound": "alu", "achieved": achieved, "peak": alu_peak_tflops, "unit": "TFLOP/s",
        "frac": achieved / alu_peak_tflops, "traffic": profiled_traffic(f"{variant}_{w.R}x{w.C}_f32"),
        "kernel": f"{variant} {w.R}x{w.C} fp32", "peak_source": (
            f"derived: {props.multi_processor_count} SMs x {FP32_LANES_PER_SM} FP32 lanes x 2 flop x "
            f"{pk.get('sm_max_mhz', 2070.0)} MHz ({pk['source']} max clock)"),
        "hbm_frac": (nbytes[dom] / (kern_ms[dom] * 1e-3) / 1e9) / float(pk["hbm_gbs"]),
    }
    if w.R == 1 and variant == "xstage":
        # a one-row block reuses no X value across outputs: every FMA needs one
        # 4-byte shared-memory load, and shared memory serves 128 bytes per
        # clock per SM, so such a kernel cannot exceed 32 FMA per clock per SM
        smem_tflops = props.multi_processor_count * 32 * 2 * float(pk.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
        roofline["smem_ceiling"] = {
            "peak": smem_tflops, "unit": "TFLOP/s", "frac": achieved / smem_tflops,
            "source": f"derived: {props.multi_processor_count} SMs x 32 fp32 shared loads/clock x 2 flop x "
                      f"{pk.get('sm_max_mhz', 2070.0)} MHz (one load per FMA)"}
    per_shape = {f"{wl.weights[i].R}x{wl.weights[i].C}": {
        "us": round(kern_ms[i] * 1e3, 2), "gflops": round(flops[i] / (kern_ms[i] * 1e-3) / 1e9, 1),
        "gbs": round(nbytes[i] / (kern_ms[i] * 1e-3) / 1e9, 1), "variant": scheds[i]["variant"],
        "frac_alu": round(flops[i] / (kern_ms[i] * 1e-3) / 1e12 / alu_peak_tflops, 4)} for i in range(nshape)}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        bsrs = [oracle.bsr_from_dense(w.W, w.R, w.C) for w in wl.weights]
        f, t, reps = time_oracle(wl, bsrs, X_np, args.cpu_seconds)
        cpu = {"value": f / t / 1e9, "unit": "GFLOP/s", "cores": 1, "kind": "oracle",
               "sample": f"full step (all 8 shapes, {N} tokens) x {reps}, fp64 accumulate, single thread"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": world, "steps": K,
            "warmup": max(args.warmup, 3), "ms_per_step": total_ms / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": WORKLOAD, "N": N, "M": 768, "K": 768, "sparsity": 80,
                       "shapes": [f"{w.R}x{w.C}" for w in wl.weights],
                       "l2": "flushed before every timed step (512 MiB write, untimed)",
                       "parallelism": f"replicas x{world}" if world > 1 else "1 GPU"},
            "gbs": gbs, "gpu_launches": launches_per_step * K,
            "clocks": clocks.summary(),
            "e2e": ({"value": e2e_value, "unit": "GFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
                    if e2e_value is not None else None),
            "roofline": roofline,
            "cpu_baseline": cpu,
            "per_shape": per_shape,
        }
        print(json.dumps(line), flush=True)
    for h in handles:
        h.destroy()


REPORT_VARIANTS = {
    1: [(None, None)],
    3: [(None, None)],
    4: [("f32", (32, 1)), ("f32", (16, 16)), ("bf16", (32, 1)), ("bf16", (16, 16))],
    5: [(None, (32, 1)), (None, (16, 16))],
}


def run_report(args):
    """One JSON line per block shape and dtype of workload 1, 3, 4 or 5."""
    import torch

    import synth
    import paper_2106_08846_gb300 as bsr
    from paper_2106_08846_gb300 import _build

    _build.build()
    bsr.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    pk = peaks()
    props = torch.cuda.get_device_properties(dev)
    mhz = float(pk.get("sm_max_mhz", 2070.0))
    fp32_peak = props.multi_processor_count * FP32_LANES_PER_SM * 2 * mhz * 1e6   # FLOP/s
    bf16_peak = float(pk["bf16_tflops"]) * 1e12
    hbm = float(pk["hbm_gbs"]) * 1e9
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def dev_array(a):
        if a.dtype == np.uint16:
            return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
        return torch.from_numpy(a).to(dev)

    for dt, shape in REPORT_VARIANTS[args.workload]:
        if args.dtype and dt is not None and dt != args.dtype:
            continue
        if args.shapes and shape is not None and f"{shape[0]}x{shape[1]}" not in args.shapes.split(","):
            continue
        only = list(range(args.weights)) if args.weights and args.workload in (3, 4) else None
        wl = synth.config(args.workload, dtype=dt, shape=shape, only=only)
        N, es = wl.N, (2 if wl.dtype == "bf16" else 4)
        X = dev_array(wl.make_X())
        handles, biases, flops, nbytes, roof_s = [], [], [], [], []
        peak = bf16_peak if wl.dtype == "bf16" else fp32_peak
        for w in wl.weights:
            arrays = bsr.bsr_from_dense(dev_array(w.W), w.R, w.C, 0.0)
            h = bsr.bsr_create(*arrays, w.R, w.C, w.M, w.K)
            h.reserve(N)
            handles.append(h)
            biases.append(torch.from_numpy(w.bias).to(dev))
            flops.append(2 * N * w.nnz)
            nbytes.append(workload_bytes(w, N, es))
            roof_s.append(max(flops[-1] / peak, nbytes[-1] / hbm))
        Y = torch.empty((N, wl.weights[0].M), dtype=X.dtype, device=dev)   # every weight of a workload is M x K
        scheds = [h.schedule() for h in handles]

        def step():
            for h, b in zip(handles, biases):
                bsr.bsr_spmm(h, X, b, Y, N, stream)

        for _ in range(max(args.warmup, 3)):
            flush.zero_()
            step()
        torch.cuda.synchronize()
        # at least about 0.4 s of timed steps, so that the clock sampler (50 ms
        # period) sees the region
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        torch.cuda.synchronize()
        K = max(1, args.steps, int(0.4 / max(e0.elapsed_time(e1) * 1e-3, 1e-6)))
        st = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
        with ClockSampler(0) as clocks:
            for k in range(K):
                flush.zero_()
                st[k][0].record(stream)
                step()
                st[k][1].record(stream)
            torch.cuda.synchronize()
        step_s = statistics.median(a.elapsed_time(b) for a, b in st) * 1e-3
        # host time to enqueue one step as separate calls
        t0 = time.perf_counter()
        step()
        host_calls_s = time.perf_counter() - t0
        torch.cuda.synchronize()
        plans = {}
        if len(handles) > 1:
            # the same step as one captured plan: the call sequence kept, and
            # (the products being independent) regrouped and fused
            for key, indep in (("plan_sequence", False), ("plan_fused", True)):
                plan = bsr.bsr_plan_create(handles, [X] * len(handles), biases, [Y] * len(handles) if not indep else
                                           [torch.empty_like(Y) for _ in handles], independent=indep)
                for _ in range(3):
                    flush.zero_()
                    plan.launch(stream)
                torch.cuda.synchronize()
                pe = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
                for k in range(K):
                    flush.zero_()
                    pe[k][0].record(stream)
                    plan.launch(stream)
                    pe[k][1].record(stream)
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                plan.launch(stream)
                host_s = time.perf_counter() - t0
                torch.cuda.synchronize()
                order, call, n_kernels = plan.order()
                plans[key] = {"us_per_step": statistics.median(a.elapsed_time(b) for a, b in pe) * 1e3,
                              "library_calls": len(set(call)), "kernels": n_kernels, "host_us": host_s * 1e6}
                plan.destroy()
        for h in handles:
            if h.check_device_status() != 0:
                raise RuntimeError("device status error during the report")
        variants = sorted({sc["variant"] + (f" (exec {sc['exec_R']}x{sc['exec_C']})"
                                             if (sc["exec_R"], sc["exec_C"]) != (sc["R"], sc["C"]) else "")
                           for sc in scheds})
        w0 = wl.weights[0]
        line = {
            "workload": args.workload, "name": wl.name, "shape": f"{w0.R}x{w0.C}", "dtype": wl.dtype, "N": N,
            "M": w0.M, "K": w0.K, "weights": len(wl.weights), "calls_per_step": len(handles),
            "variants": variants, "steps": K, "us_per_step": step_s * 1e6,
            "gflops": sum(flops) / step_s / 1e9, "gbs": sum(nbytes) / step_s / 1e9,
            "roofline": {"us_per_step": sum(roof_s) * 1e6, "frac": sum(roof_s) / step_s,
                         "bound": "bytes" if sum(b / hbm for b in nbytes) >= sum(f / peak for f in flops) else "flops",
                         "peak_tflops": peak / 1e12, "hbm_gbs": hbm / 1e9,
                         "peak_source": ("bf16 tensor, " if wl.dtype == "bf16" else "FP32 FMA, derived from ") +
                                        f"{pk['source']} peaks"},
            "host_us_per_step_calls": host_calls_s * 1e6,
            "l2": "flushed before every step", "clocks": clocks.summary(), "data": "synthetic",
        }
        line.update(plans)
        print(json.dumps(line), flush=True)
        for h in handles:
            h.destroy()


def main():
    args = parse()
    if args.workload != 2:
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
