#!/usr/bin/env python
"""Throughput of the AQ x A8 layer on GB300 (one JSON line on stdout).

Workload (default): the fused qkv projection of an LDM-4-like UNet at its 8x8
level for 32 images x CFG pair: T = 4096 tokens, K = 960, N = 2880, 2x8
codebooks (W2A8), seeded synthetic weights and activations.  One step is the
whole hot path of that layer: 8-bit activation quantization of the fp16
input, decode of the AQ weight, tensor-core contraction, fused scale/bias
epilogue to fp16.

Timing: CUDA-graph replay of 8 steps that rotate over 8 independent buffer
sets (inputs, codes, outputs: > 300 MB together, larger than the 129 MB L2),
CUDA events on the launching stream, warm-up first, barrier + synchronize on
both sides, max over ranks.  The dominant kernel (the tensor-core GEMM) is
timed by the library's own event pairs, captured as event-record nodes into a
second graph that is replayed once inside the same timed region.  `e2e` repeats the step through the public C ABI with the
input copied from pinned host memory and the output copied back every step.

--impl reference times the CPU oracle (plain numpy fp64) on the same workload.
Multi-GPU: independent replicas, one per rank (the layer needs no exchange).
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

WORKLOADS = {
    "qkv": dict(cfg=1, name="AQ linear qkv projection T=4096 K=960 N=2880 W2A8 (2x8 codebooks, g=8)"),
}
NSETS = 8

# DRAM traffic of one launch of the tensor-core GEMM kernel on this workload,
# from `ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum` (see the
# summary under profiles/), valid only for the kernel sources it was taken on.
TRAFFIC = {
    "qkv": {"bytes": None, "sources_sha": None},
}
KERNEL_SOURCES = ["paper_2506_05960_gb300/csrc/aq_gemm.cu", "paper_2506_05960_gb300/csrc/aq_ptx.cuh"]


def sources_sha() -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return dict(hbm_gbs=d["hbm_gbs"], bf16_tflops=d["bf16_tflops"],
                    bf16_tflops_sustained=d.get("bf16_tflops_sustained"), source="measured")
    return dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0, source="fallback")


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines: list[str] = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        time.sleep(0.3)      # let the first samples arrive before the timed region

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=5)
        sm, smax, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
                power.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------- workload
def make_sets(cfg: int, nsets: int):
    from aq_synth import CONFIGS, make_linear
    spec = CONFIGS[cfg]
    sets = []
    for i in range(nsets):
        inp = make_linear(spec, seed=cfg * 1000 + i)
        # fp16 activations whose 8-bit quantization with s_x gives the seeded int8 values
        inp["x16"] = (inp["xq"].astype(np.float32) * np.float32(spec.s_x)).astype(np.float16)
        sets.append(inp)
    return spec, sets


def flops_per_step(spec) -> float:
    return 2.0 * spec.T * spec.N * spec.K


def alg_bytes(spec) -> int:
    """Algorithmic bytes of the layer: codes, codebooks, int8 activations once, output,
    scale + bias (decoded weights and other scratch excluded)."""
    codes = spec.N * spec.K * spec.M * spec.B // (8 * spec.g)
    books = spec.M * (1 << spec.B) * spec.g * 2
    return codes + books + spec.T * spec.K + spec.T * spec.N * 2 + 4 * spec.N


# ----------------------------------------------------------------------------- oracle (CPU)
def time_oracle(spec, inp, min_seconds: float = 10.0, max_steps: int = 50) -> dict:
    """The oracle as it stands (float64 decode + numpy matmul) on the full layer, repeated
    until about `min_seconds` of CPU time."""
    from oracle import aq_oracle as O
    steps = 0
    t0 = time.perf_counter()
    while True:
        O.layer_f64(inp)
        steps += 1
        el = time.perf_counter() - t0
        if el >= min_seconds or steps >= max_steps:
            break
    cores = len(os.sched_getaffinity(0))
    return {"value": flops_per_step(spec) * steps / el / 1e12, "unit": "TFLOP/s",
            "cores": cores, "kind": "oracle",
            "sample": f"full layer (T={spec.T}, K={spec.K}, N={spec.N}) x {steps} step(s), "
                      f"{el:.1f} s, numpy float64 BLAS on {cores} host cores",
            "seconds": el, "steps": steps}


# ----------------------------------------------------------------------------- main
def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_reference(args, workload):
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    spec, sets = make_sets(WORKLOADS[workload]["cfg"], 1)
    inp = sets[0]
    from oracle import aq_oracle as O
    for _ in range(args.warmup):
        O.layer_f64(inp)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        O.layer_f64(inp)
        times.append(time.perf_counter() - t0)
    el = sum(times)
    val = flops_per_step(spec) * args.steps / el / 1e12
    cores = len(os.sched_getaffinity(0))
    line = {"impl": "reference", "metric": "AQ layer dense-equivalent TFLOP/s", "value": val,
            "unit": "TFLOP/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": el / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOADS[workload]["name"], "T": spec.T, "K": spec.K,
                       "N": spec.N, "M": spec.M, "B": spec.B, "g": spec.g},
            "cpu_baseline": {"value": val, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                             "sample": f"full layer per step, {args.steps} steps"},
            "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="qkv", choices=sorted(WORKLOADS))
    ap.add_argument("--e2e-steps", type=int, default=100)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    if args.impl == "reference":
        return run_reference(args, args.workload)

    world, rank, local = dist_setup()
    spec, sets = make_sets(WORKLOADS[args.workload]["cfg"], NSETS)

    # CPU baseline first (before any GPU work), rank 0 at N=1 only
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = time_oracle(spec, sets[0], min_seconds=args.cpu_seconds)

    import torch
    import paper_2506_05960_gb300 as aq

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    aq.load_library()

    T, K, N, g, M, B = spec.T, spec.K, spec.N, spec.g, spec.M, spec.B
    ws_bytes = aq.aq_linear_workspace_size(T, K, N, g, M, B)
    bufs = []
    for inp in sets:
        b = {}
        b["x16"] = torch.from_numpy(inp["x16"]).to(dev)
        codes = torch.from_numpy(inp["codes"]).to(dev)
        b["packed"] = torch.empty(aq.aq_packed_size(N, K, g, M, B), dtype=torch.uint8, device=dev)
        aq.aq_pack(codes, b["packed"], N, K, g, M, B)
        b["books"] = torch.from_numpy(inp["codebooks"]).to(dev)
        b["scale"] = torch.from_numpy(inp["scale"]).to(dev)
        b["bias"] = torch.from_numpy(inp["bias"]).to(dev)
        b["xq"] = torch.empty((T, K), dtype=torch.int8, device=dev)
        b["y"] = torch.empty((T, N), dtype=torch.float16, device=dev)
        b["ws"] = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device=dev)
        bufs.append(b)
    torch.cuda.synchronize()
    s_x = spec.s_x
    stream = torch.cuda.Stream(device=dev)

    def step(b, st):
        aq.aq_quant_act(b["x16"], b["xq"], T * K, s_x, stream=st)
        aq.aq_linear(b["xq"], s_x, b["packed"], b["books"], b["scale"], b["bias"], b["y"],
                     aq.AQ_DTYPE_F16, T, K, N, g, M, B, b["ws"], ws_bytes, stream=st)

    # warm-up (eager); one pass with kernel timing on fills the library's event pool so
    # that capture below needs no event creation
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            step(bufs[i % NSETS], stream)
        aq.aq_profile_enable(True)
        for i in range(2 * NSETS):
            step(bufs[i % NSETS], stream)
    stream.synchronize()
    aq.aq_profile_read()
    aq.aq_profile_enable(False)
    assert aq.aq_device_error() == 0

    # capture the main graph (NSETS steps, one per buffer set) and a copy whose library
    # calls carry event-record nodes around every kernel (for per-kernel device time)
    g_main = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_main, stream=stream):
        for i in range(NSETS):
            step(bufs[i], stream)
    aq.aq_profile_enable(True)
    g_prof = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_prof, stream=stream):
        for i in range(NSETS):
            step(bufs[i], stream)
    for _ in range(2):
        g_main.replay()
    stream.synchronize()

    reps = max(1, args.steps // NSETS)
    steps = reps * NSETS
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    sampler.start()
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        ev0.record(stream)
        for _ in range(reps):
            g_main.replay()
        ev1.record(stream)
        g_prof.replay()          # per-kernel event pairs (read below)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    clocks = sampler.stop()
    ms_total = ev0.elapsed_time(ev1)
    prof = aq.aq_profile_read()
    aq.aq_profile_enable(False)
    assert aq.aq_device_error() == 0
    if pg:
        t = torch.tensor([ms_total], dtype=torch.float64, device=dev)
        pg.all_reduce(t, op=pg.ReduceOp.MAX)
        ms_total = float(t.item())
    ms_step = ms_total / steps
    fl = flops_per_step(spec)
    value = world * fl / (ms_step * 1e-3) / 1e12

    gemm_ms, gemm_n = prof["gemm"]
    gemm_avg_ms = gemm_ms / gemm_n if gemm_n else float("nan")
    peaks = measured_peaks()
    achieved = fl / (gemm_avg_ms * 1e-3) / 1e12
    tr = TRAFFIC.get(args.workload, {})
    traffic = tr.get("bytes") if tr.get("sources_sha") == sources_sha() else None
    launches_per_step = sum(n for k, (ms, n) in prof.items()) / NSETS

    # e2e through the public API: pinned host input -> device, step, device -> pinned host
    h_x = [torch.from_numpy(inp["x16"]).pin_memory() for inp in sets[:2]]
    h_y = torch.empty((T, N), dtype=torch.float16).pin_memory()
    e2e_steps = max(1, args.e2e_steps)
    with torch.cuda.stream(stream):
        for i in range(3):
            b = bufs[i % 2]
            b["x16"].copy_(h_x[i % 2], non_blocking=True)
            step(b, stream)
            h_y.copy_(b["y"], non_blocking=True)
        stream.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(e2e_steps):
            b = bufs[i % 2]
            b["x16"].copy_(h_x[i % 2], non_blocking=True)
            step(b, stream)
            h_y.copy_(b["y"], non_blocking=True)
        e1.record(stream)
    stream.synchronize()
    e2e_ms = e0.elapsed_time(e1) / e2e_steps
    if pg:
        t = torch.tensor([e2e_ms], dtype=torch.float64, device=dev)
        pg.all_reduce(t, op=pg.ReduceOp.MAX)
        e2e_ms = float(t.item())

    if rank == 0:
        line = {
            "metric": "AQ layer dense-equivalent TFLOP/s (2*T*N*K / step time)",
            "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
            "config": {"workload": WORKLOADS[args.workload]["name"], "T": T, "K": K, "N": N,
                       "g": g, "M": M, "B": B, "parallelism": f"replicas{world}",
                       "l2": f"inputs larger than L2: {NSETS} rotating buffer sets",
                       "timing": "CUDA graph replay of 8 steps, CUDA events"},
            "hbm_gbs_algorithmic": alg_bytes(spec) / (ms_step * 1e-3) / 1e9,
            "roofline": {"bound": "tensor", "kernel": "aq_gemm_kernel", "achieved": achieved,
                         "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": achieved / peaks["bf16_tflops"], "traffic": traffic,
                         "peak_source": f"{peaks['source']} bf16 burst (fp16 dense rate is equal)",
                         "frac_of_sustained": (achieved / peaks["bf16_tflops_sustained"]
                                               if peaks.get("bf16_tflops_sustained") else None),
                         "kernel_ms": gemm_avg_ms},
            "kernel_ms": {k: (ms / n if n else None) for k, (ms, n) in prof.items()},
            "step_roofline_frac": (max(fl / (peaks["bf16_tflops"] * 1e12),
                                       alg_bytes(spec) / (peaks["hbm_gbs"] * 1e9)) / (ms_step * 1e-3)),
            "cpu_baseline": cpu and {k: cpu[k] for k in ("value", "unit", "cores", "kind", "sample")},
            "e2e": {"value": world * fl / (e2e_ms * 1e-3) / 1e12, "unit": "TFLOP/s",
                    "ms_per_step": e2e_ms, "h2d_bytes_per_step": T * K * 2,
                    "d2h_bytes_per_step": T * N * 2},
            "gpu_launches": int(round(launches_per_step * steps)) + sum(n for _, n in prof.values()),
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    if pg:
        pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
