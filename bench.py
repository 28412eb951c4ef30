#!/usr/bin/env python
"""Throughput of the AQ x A8 layer on GB300 (one JSON line on stdout).

Headline workload: the fused qkv projection of an LDM-4-like UNet at its 8x8
level for 32 images x CFG pair: T = 4096 tokens, K = 960, N = 2880, 2x8
codebooks (W2A8), seeded synthetic weights and activations.  One step is the
whole hot path of that layer through the C ABI (aq_linear_f16): 8-bit
quantization of the fp16 input, decode of the AQ weight, tensor-core
contraction, fused scale/bias epilogue to fp16.

Timing: exactly --steps steps, as CUDA-graph replays of 8 steps that rotate
over 8 independent buffer sets (inputs, codes, outputs: > 300 MB together,
larger than the 129 MB L2) plus one graph of the remaining steps, CUDA events
on the launching stream, warm-up first, barrier + synchronize on both sides,
max over ranks.  The dominant kernel (the tensor-core GEMM) is timed by itself
right after: a graph of 8 GEMM launches on the same buffer sets (weights
decoded beforehand, AQ_PATH_PREDECODED through aq_linear_a16), replayed at
least 50 times and for at least 20 ms; the library's per-kernel event pairs
(aq_profile_*) over plain launches of the step are reported beside it.
`e2e` repeats the step through the C ABI with every step's fp16 input copied from
pinned host memory and its fp16 output copied back: copy-in, compute and
copy-out on three streams, so one step's compute overlaps the neighbouring
steps' copies (the serial single-stream figure is reported beside it).  A
cuBLAS fp16 GEMM of the same shapes is timed as context for the GEMM's
roofline fraction.  `layers` times the other
workloads (64x64 W4A8 conv, 8x8 conv with one 2^16-entry codebook) and
`unet_forward` one UNet-shaped forward (97 AQ layers, W2A8 and W4A8, batches 2, 16
and 64), with each layer preceded by the quantizer, or writing the next layer's
int8 activations from its epilogue.  A small-T sweep (T = 1..64) times every path.

--impl reference times the CPU oracle (numpy float64) on the headline workload.
`cpu_baselines` times the oracle on every workload (single-threaded and on all host
cores), in child processes started before any GPU work.
Multi-GPU: independent replicas, one per rank (the layer has no exchange step).
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

HEADLINE = "AQ linear qkv projection T=4096 K=960 N=2880 W2A8 (2x8 codebooks, g=8)"
METRIC = "AQ layer dense-equivalent TFLOP/s (2*T*N*K / step time)"
NSETS = 8

# DRAM traffic of one launch of the tensor-core GEMM on the headline workload, from an ncu
# capture of one launch (dram__bytes_read.sum + dram__bytes_write.sum; summary in
# profiles/aq_gemm_kernel_a16_qkv_T4096_K960_N2880.md); reported only while the kernel sources
# hash to the ones it was captured on (the key is refreshed either by a new capture or, after
# changes elsewhere in these files, once the GEMM kernels' code sections hash the same).
KERNEL_SOURCES = ["paper_2506_05960_gb300/csrc/aq_gemm.cu", "paper_2506_05960_gb300/csrc/aq_ptx.cuh",
                  "paper_2506_05960_gb300/csrc/aq_quant.cuh", "paper_2506_05960_gb300/csrc/aq_internal.h"]
TRAFFIC = {"bytes": 13476352, "sources_sha": "49f7b985b8b5ad4a"}


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
def headline_sets(nsets: int):
    from aq_synth import WORKLOADS, make_linear
    spec = WORKLOADS["qkv"]
    return spec, [make_linear(spec, seed=1000 + i) for i in range(nsets)]


def linear_flops(T, N, K) -> float:
    return 2.0 * T * N * K


def alg_bytes(T, K, N, M, B, g=8, out_bytes=2) -> int:
    """Algorithmic bytes of one layer: codes, codebooks, int8 activations once, output,
    scale + bias (decoded weights and scratch excluded)."""
    return N * K * M * B // (8 * g) + M * (1 << B) * g * 2 + T * K + T * N * out_bytes + 4 * N


# ----------------------------------------------------------------------------- oracle (CPU)
def time_oracle(inp, flops, min_seconds: float = 10.0, max_steps: int = 50) -> dict:
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
    spec = inp["spec"]
    return {"value": flops * steps / el / 1e12, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
            "sample": f"full layer (T={spec.T}, K={spec.K}, N={spec.N}) x {steps} step(s), "
                      f"{el:.1f} s, numpy float64 BLAS on {cores} host cores"}


def oracle_workloads(mode: str):
    """(name, layer dicts, GFLOP) per workload timed by the CPU oracle.  mode "single":
    configs 0-3 (tiny linear, qkv, 64x64 W4A8 conv, 8x8 conv with a 2^16 book); "all":
    configs 1-3 and the UNet-shaped forward (97 layers, W2A8, batch 2)."""
    from aq_synth import (ConvSpec, LinearSpec, SEEDS, WORKLOADS, make_conv, make_linear,
                          unet_sweep_layers)
    out = []
    names = (["tiny_linear"] if mode == "single" else []) + ["qkv", "conv64", "conv8_book16"]
    for name in names:
        spec = WORKLOADS[name]
        inp = (make_conv if isinstance(spec, ConvSpec) else make_linear)(spec, seed=SEEDS[name])
        out.append((name, [inp], linear_flops(spec.T, spec.N if isinstance(spec, LinearSpec)
                                              else spec.Cout, spec.K) / 1e9))
    if mode == "all":
        layers, gflop, seed = [], 0.0, 4200
        for kind, res, cin, cout, stride, count in unet_sweep_layers():
            for _ in range(count):
                seed += 1
                if kind == "conv3":
                    spec = ConvSpec(Nb=2, H=res * stride, W=res * stride, Cin=cin, Cout=cout,
                                    stride=stride, M=2, B=8, cb_std=0.03)
                    layers.append(make_conv(spec, seed))
                    gflop += linear_flops(spec.T, cout, spec.K) / 1e9
                else:
                    spec = LinearSpec(T=2 * res * res, K=cin, N=cout, M=2, B=8, cb_std=0.03,
                                      act="normal40")
                    layers.append(make_linear(spec, seed))
                    gflop += linear_flops(spec.T, cout, cin) / 1e9
        out.append(("unet_w2a8_batch2", layers, gflop))
    return out


def cpu_oracle_child(mode: str, seconds: float) -> None:
    """Child process of run_cpu_baselines: time the oracle (decode in float64, then the
    float64 matmul / convolution) on each workload and print one JSON object."""
    from oracle import aq_oracle as O
    res = {}
    for name, layers, gflop in oracle_workloads(mode):
        reps, el = 0, 0.0
        while reps < 1 or (el < seconds and reps < 20):
            t0 = time.perf_counter()
            for inp in layers:
                O.layer_f64(inp)
            el += time.perf_counter() - t0
            reps += 1
        res[name] = {"ms_per_pass": el / reps * 1e3, "gflop": gflop,
                     "tflops": gflop * reps / el / 1e3, "passes": reps}
    print(json.dumps(res), flush=True)


def run_cpu_baselines(seconds: float = 1.0) -> dict:
    """The oracle as it stands on every workload, single-threaded (BLAS/OpenMP threads = 1)
    for configs 0-3 and on all host cores for configs 1-4, each in a child process (started
    before any GPU work).  The UNet forward at batch 16 and 64 is extrapolated linearly from
    batch 2 (the oracle's work is linear in the batch) and labelled so."""
    cores = len(os.sched_getaffinity(0))
    out = {"kind": "oracle", "cores": cores}
    for mode in ("single", "all"):
        env = dict(os.environ)
        n = "1" if mode == "single" else str(cores)
        for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
            env[v] = n
        try:
            r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-oracle", mode,
                                "--cpu-seconds", str(seconds)], env=env, capture_output=True,
                               text=True, timeout=600)
            vals = json.loads(r.stdout.strip().splitlines()[-1])
        except Exception as e:  # reported, not fatal: the GPU line is the product
            out[mode] = {"error": f"{type(e).__name__}: {e}"[:300]}
            continue
        if mode == "all" and "unet_w2a8_batch2" in vals:
            b2 = vals["unet_w2a8_batch2"]
            for batch in (16, 64):
                f = batch / 2
                vals[f"unet_w2a8_batch{batch}"] = {
                    "ms_per_pass": b2["ms_per_pass"] * f, "gflop": b2["gflop"] * f,
                    "tflops": b2["tflops"], "extrapolated_from": "batch 2 (linear in batch)"}
        out[mode] = dict(vals, threads=int(n))
    return out


def max_over_ranks(dist, value: float, device) -> float:
    """The largest `value` over all ranks of the process group (every rank receives it):
    the job takes as long as its slowest replica."""
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, flops_per_step: float, ms_per_step: float) -> float:
    """Whole-job dense-equivalent TFLOP/s: every rank runs its own replica of the step
    (weak scaling), so the job does `world` steps in the slowest rank's step time."""
    return world * flops_per_step / (ms_per_step * 1e-3) / 1e12


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_reference(args):
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    spec, sets = headline_sets(1)
    inp = sets[0]
    from oracle import aq_oracle as O
    # each step is a bounded sample of the layer: the first Ts tokens, Ts sized so the
    # whole --warmup + --steps run takes about two minutes
    t0 = time.perf_counter()
    O.layer_f64(inp)
    full_s = time.perf_counter() - t0
    budget = 120.0 / max(1, args.steps + args.warmup)
    Ts = int(min(spec.T, max(16, spec.T * budget / max(full_s, 1e-6))))
    sample = dict(inp)
    sample["xq"] = inp["xq"][:Ts]
    for _ in range(args.warmup):
        O.layer_f64(sample)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        O.layer_f64(sample)
        times.append(time.perf_counter() - t0)
    el = sum(times)
    val = linear_flops(Ts, spec.N, spec.K) * args.steps / el / 1e12
    cores = len(os.sched_getaffinity(0))
    line = {"impl": "reference", "metric": METRIC, "value": val,
            "unit": "TFLOP/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": el / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": HEADLINE, "T": spec.T, "K": spec.K, "N": spec.N, "M": spec.M,
                       "B": spec.B, "g": spec.g},
            "cpu_baseline": {"value": val, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                             "sample": f"first {Ts} of {spec.T} tokens of the layer per step "
                                       f"(full decode), {args.steps} steps"},
            "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- GPU helpers
class Dev:
    """Device copies of one seeded layer plus its output and workspace; step() is one pass
    of the hot path through the C ABI (quantizer, then the layer on the AUTO path)."""

    def __init__(self, aq, torch, inp, dev, path=0, xq_dev=None):
        """xq_dev: int8 activations already on the device (shape of the layer's input),
        used instead of inp["xq"] for large batches (inp then only supplies weights)."""
        self.aq, self.torch = aq, torch
        s = inp["spec"]
        self.spec = s
        self.conv = inp["xq"].ndim == 4
        N, G, M = inp["codes"].shape
        K = G * 8
        B = 8 if inp["codes"].dtype == np.uint8 else 16
        self.N, self.K, self.M, self.B, self.path = N, K, M, B, path

        def t(a):
            return torch.from_numpy(np.ascontiguousarray(a)).to(dev)

        codes = t(inp["codes"])
        self.packed = torch.empty(aq.aq_packed_size(N, K, 8, M, B), dtype=torch.uint8, device=dev)
        aq.aq_pack(codes, self.packed, N, K, 8, M, B)
        self.books, self.scale, self.bias = t(inp["codebooks"]), t(inp["scale"]), t(inp["bias"])
        # fp16 activations whose 8-bit quantization with s_x gives the seeded int8 values
        if xq_dev is None:
            x16 = (inp["xq"].astype(np.float32) * np.float32(inp["s_x"])).astype(np.float16)
            self.x16 = t(x16)
        else:
            self.x16 = (xq_dev.float() * float(np.float32(inp["s_x"]))).half()
        self.xq = torch.empty(tuple(self.x16.shape), dtype=torch.int8, device=dev)
        self.s_x = inp["s_x"]
        self.yq = None
        if self.conv:
            self.T = s.Nb * s.Ho * s.Wo
            self.ws_bytes = aq.aq_conv2d_workspace_size(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3,
                                                        s.stride, 1, 8, M, B, path)
            self.y = torch.empty((s.Nb, s.Ho, s.Wo, N), dtype=torch.float16, device=dev)
        else:
            self.T = self.x16.shape[0]
            self.ws_bytes = aq.aq_linear_workspace_size(self.T, K, N, 8, M, B, path)
            self.y = torch.empty((self.T, N), dtype=torch.float16, device=dev)
            self.ws16_bytes = aq.aq_linear_f16_workspace_size(self.T, K, N, 8, M, B, path)
            self.ws16 = None
        self.ws = torch.empty(max(self.ws_bytes, 16), dtype=torch.uint8, device=dev)
        self.flops = linear_flops(self.T, N, K)

    def quant(self, st):
        self.aq.aq_quant_act(self.x16, self.xq, self.xq.numel(), self.s_x, stream=st)

    def layer(self, st):
        aq, s = self.aq, self.spec
        if self.conv:
            aq.aq_conv2d_nhwc(self.xq, self.s_x, self.packed, self.books, self.scale, self.bias,
                              self.y, aq.AQ_DTYPE_F16, s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3,
                              s.stride, 1, 8, self.M, self.B, self.ws, self.ws_bytes, self.path,
                              stream=st)
        else:
            aq.aq_linear(self.xq, self.s_x, self.packed, self.books, self.scale, self.bias, self.y,
                         aq.AQ_DTYPE_F16, self.T, self.K, self.N, 8, self.M, self.B, self.ws,
                         self.ws_bytes, self.path, stream=st)

    def layer_q8(self, st, s_out=0.02, path=None, ws=None):
        """The layer with the next layer's quantizer in its epilogue (int8 output); `ws`
        replaces the layer's workspace (e.g. one holding weights decoded beforehand)."""
        aq, s = self.aq, self.spec
        path = self.path if path is None else path
        ws_t = self.ws if ws is None else ws
        if self.yq is None:
            self.yq = self.torch.empty(tuple(self.y.shape), dtype=self.torch.int8,
                                       device=self.y.device)
        if self.conv:
            aq.aq_conv2d_nhwc_q8(self.xq, self.s_x, self.packed, self.books, self.scale,
                                 self.bias, self.yq, s_out, s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3,
                                 s.stride, 1, 8, self.M, self.B, ws_t, ws_t.numel(),
                                 path, stream=st)
        else:
            aq.aq_linear_q8(self.xq, self.s_x, self.packed, self.books, self.scale, self.bias,
                            self.yq, s_out, self.T, self.K, self.N, 8, self.M, self.B, ws_t,
                            ws_t.numel(), path, stream=st)

    def layer_ex(self, st, path=None, ws=None, s_out=0.02):
        """The layer through aq_*_ex: activations in self.in_kind (int8 codes self.xq, or fp16
        codes self.xh), output in self.out_kind (the next layer's codes, scale s_out) into
        self.yc; `ws` replaces the layer's workspace (e.g. one holding decoded weights)."""
        aq, s = self.aq, self.spec
        path = self.path if path is None else path
        ws_t = self.ws if ws is None else ws
        act = self.xh if self.in_kind == aq.AQ_DTYPE_F16_CODES else self.xq
        if self.conv:
            aq.aq_conv2d_nhwc_ex(act, self.in_kind, self.s_x, self.packed, self.books, self.scale,
                                 self.bias, self.yc, self.out_kind, s_out, s.Nb, s.H, s.W, s.Cin,
                                 s.Cout, 3, 3, s.stride, 1, 8, self.M, self.B, ws_t, ws_t.numel(),
                                 path, stream=st)
        else:
            aq.aq_linear_ex(act, self.in_kind, self.s_x, self.packed, self.books, self.scale,
                            self.bias, self.yc, self.out_kind, s_out, self.T, self.K, self.N, 8,
                            self.M, self.B, ws_t, ws_t.numel(), path, stream=st)

    def gemm_a16(self, st, xh, ws):
        """The tensor-core GEMM alone: fp16 activations xh (the 8-bit codes as fp16 values) and
        weights decoded beforehand into ws (AQ_PATH_PREDECODED)."""
        self.aq.aq_linear_a16(xh, self.s_x, self.packed, self.books, self.scale, self.bias,
                              self.y, self.aq.AQ_DTYPE_F16, self.T, self.K, self.N, 8, self.M,
                              self.B, ws, ws.numel(), self.aq.AQ_PATH_PREDECODED, stream=st)

    def decode_only(self, st, wbuf):
        self.aq.aq_decode(self.packed, self.books, wbuf, self.N, self.K, 8, self.M, self.B,
                          stream=st)

    def step(self, st):
        self.quant(st)
        self.layer(st)

    def step_f16(self, st):
        """The same pass from the fp16 activations in one call (aq_linear_f16)."""
        if self.ws16 is None:
            self.ws16 = self.torch.empty(self.ws16_bytes, dtype=self.torch.uint8,
                                         device=self.y.device)
        self.aq.aq_linear_f16(self.x16, self.s_x, self.packed, self.books, self.scale, self.bias,
                              self.y, self.aq.AQ_DTYPE_F16, self.T, self.K, self.N, 8, self.M,
                              self.B, self.ws16, self.ws16_bytes, self.path, stream=st)


def capture(torch, stream, fn):
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    return g


def replay_ms(torch, stream, g, reps):
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        g.replay()
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / reps


def unet_forward(aq, torch, dev, stream, M, batch=2, reps=20, fused_quant=False,
                 decode_ahead=False, mixed=False):
    """One UNet-shaped forward: every AQ layer of the LDM-4-like sweep, captured as one
    graph.  Each layer is preceded by its activation quantizer (aq_quant_act), or, with
    fused_quant, writes int8 output through its _q8 epilogue instead (the chain of
    layers then has no separate quantizer pass).  With mixed (and fused_quant), each layer
    takes its activations in the form its own plan reads faster -- the codes as fp16 values
    where the shared-memory A form wins (aq_*_f16_plan), else int8 -- and the layer before it
    writes that form (aq_*_ex).  Above batch 2 the int8 activations are drawn on the device
    (seeded torch generator) and the host arrays only supply the weights.
    Returns (ms, GFLOP, layers)."""
    from aq_synth import ConvSpec, LinearSpec, make_conv, make_linear, unet_sweep_layers
    layers = []
    seed = 4000 + 100 * M
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed + batch)
    big = batch > 2

    def acts(shape):
        # round(N(0, 40)) clipped to +-127, as the host generator's "normal40"
        v = torch.randn(shape, generator=gen, device=dev) * 40.0
        return v.round().clamp_(-127, 127).to(torch.int8)

    for kind, res, cin, cout, stride, count in unet_sweep_layers():
        for _ in range(count):
            seed += 1
            if kind == "conv3":
                spec = ConvSpec(Nb=batch, H=res * stride, W=res * stride, Cin=cin, Cout=cout,
                                stride=stride, M=M, B=8, cb_std=0.03)
                if big:
                    wspec = ConvSpec(Nb=1, H=8, W=8, Cin=cin, Cout=cout, M=M, B=8, cb_std=0.03)
                    inp = dict(make_conv(wspec, seed), spec=spec)
                    xq = acts((batch, res * stride, res * stride, cin))
                    layers.append(Dev(aq, torch, inp, dev, xq_dev=xq))
                else:
                    layers.append(Dev(aq, torch, make_conv(spec, seed), dev))
            else:
                T = batch * res * res
                spec = LinearSpec(T=T, K=cin, N=cout, M=M, B=8, cb_std=0.03, act="normal40")
                if big:
                    wspec = LinearSpec(T=16, K=cin, N=cout, M=M, B=8, cb_std=0.03, act="normal40")
                    inp = dict(make_linear(wspec, seed), spec=spec)
                    layers.append(Dev(aq, torch, inp, dev, xq_dev=acts((T, cin))))
                else:
                    layers.append(Dev(aq, torch, make_linear(spec, seed), dev))
    torch.cuda.synchronize()

    # decode_ahead (with fused_quant): the dense-path layers -- and, with 4 or more
    # codebooks, also the token-poor ones that AUTO sends down the fused path -- take
    # AQ_PATH_PREDECODED, and a second stream decodes those layers' weights (aq_decode into
    # a workspace) ahead of the layer chain; each layer waits only for its own decode.
    # (Measured at batch 2: predecoding the fused-path layers too took the W4A8 forward from
    # 1.457 to 1.408 ms but the W2A8 one from 1.288 to 1.359 ms -- with two codebooks the
    # in-GEMM decode costs less than streaming the 8x larger decoded weights.)
    # Every weight is still decoded once per forward; each such layer then needs its decoded
    # weights resident until it runs (here: one workspace per layer).
    side = torch.cuda.Stream(device=dev) if decode_ahead else None
    F16C, I8 = aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_I8
    for i, L in enumerate(layers):
        L.in_kind = I8
        if mixed:
            s = L.spec
            pf = (aq.aq_conv2d_f16_plan(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, 1, 8, L.M,
                                        L.B, L.path) if L.conv
                  else aq.aq_linear_f16_plan(L.T, L.K, L.N, 8, L.M, L.B, L.path))
            L.in_kind = F16C if pf["a16"] else I8
    for i, L in enumerate(layers):
        L.out_kind = layers[i + 1].in_kind if i + 1 < len(layers) else I8
        if mixed:
            L.yc = torch.empty(tuple(L.y.shape),
                               dtype=torch.float16 if L.out_kind == F16C else torch.int8,
                               device=dev)
            if L.in_kind == F16C:
                s = L.spec
                nb = (aq.aq_conv2d_ex_workspace_size(F16C, s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3,
                                                     s.stride, 1, 8, L.M, L.B, L.path)
                      if L.conv else
                      aq.aq_linear_ex_workspace_size(F16C, L.T, L.K, L.N, 8, L.M, L.B, L.path))
                if nb > L.ws.numel():
                    L.ws = torch.empty(nb, dtype=torch.uint8, device=dev)
    for L in layers:
        L.dense = False
        L.ws_pre = L.ws
        if decode_ahead:
            s = L.spec
            plan = (aq.aq_conv2d_plan(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, 1, 8, L.M,
                                      L.B, L.path) if L.conv
                    else aq.aq_linear_plan(L.T, L.K, L.N, 8, L.M, L.B, L.path))
            L.dense = plan["path"] == aq.AQ_PATH_DENSE
            if L.M >= 4 and not L.dense:
                L.dense = True
                nb = (aq.aq_conv2d_workspace_size(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride,
                                                  1, 8, L.M, L.B, aq.AQ_PATH_PREDECODED)
                      if L.conv else
                      aq.aq_linear_workspace_size(L.T, L.K, L.N, 8, L.M, L.B,
                                                  aq.AQ_PATH_PREDECODED))
                L.ws_pre = torch.empty(nb, dtype=torch.uint8, device=dev)
            if L.dense and L.in_kind == F16C:
                # the fp16-code form's plan may split K differently: room for its partials too
                nb16 = (aq.aq_conv2d_ex_workspace_size(F16C, s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3,
                                                       s.stride, 1, 8, L.M, L.B,
                                                       aq.AQ_PATH_PREDECODED)
                        if L.conv else
                        aq.aq_linear_ex_workspace_size(F16C, L.T, L.K, L.N, 8, L.M, L.B,
                                                       aq.AQ_PATH_PREDECODED))
                if nb16 > L.ws_pre.numel():
                    L.ws_pre = torch.empty(nb16, dtype=torch.uint8, device=dev)

    def fwd():
        if decode_ahead:
            start = torch.cuda.Event()
            start.record(stream)
            side.wait_event(start)
            ready = []
            for L in layers:
                if L.dense:
                    aq.aq_decode(L.packed, L.books, L.ws_pre, L.N, L.K, 8, L.M, L.B, stream=side)
                    e = torch.cuda.Event()
                    e.record(side)
                    ready.append(e)
                else:
                    ready.append(None)
            for L, e in zip(layers, ready):
                if e is not None:
                    stream.wait_event(e)
                if mixed:
                    L.layer_ex(stream, path=aq.AQ_PATH_PREDECODED if L.dense else None,
                               ws=L.ws_pre)
                else:
                    L.layer_q8(stream, path=aq.AQ_PATH_PREDECODED if L.dense else None,
                               ws=L.ws_pre)
            return
        for L in layers:
            if mixed:
                L.layer_ex(stream)
            elif fused_quant:
                L.layer_q8(stream)
            else:
                L.step(stream)

    with torch.cuda.stream(stream):
        for L in layers:
            L.quant(stream)          # int8 inputs for the fused-quantizer chain
            if L.in_kind == F16C:
                L.xh = L.xq.to(torch.float16)   # the same codes as fp16 values
        for _ in range(2):
            fwd()
    stream.synchronize()
    g = capture(torch, stream, fwd)
    ms = replay_ms(torch, stream, g, reps)
    gflop = sum(L.flops for L in layers) / 1e9
    del g
    return ms, gflop, len(layers)


KERNEL_WORKLOADS = {
    "quant": "aq_quant_act on the qkv input (4096 x 960 fp16)",
    "decode": "aq_decode of the qkv weight (2880 x 960, 2x8)",
    "linear_f16": "aq_linear_f16 on the qkv layer (quantizer, decode, GEMM)",
    "gemm_a16": ("aq_linear_a16 on the qkv layer, weights decoded beforehand (the tensor-core "
                 "GEMM alone, fp16 activation codes)"),
    "fused128": "aq_linear, T=128 K=960 N=2880 2x8 (fused decode, K split in cluster)",
    "few4": "aq_linear, T=4 K=960 N=2880 2x8 (few-token kernel)",
    "lut8": "aq_linear, T=8 K=960 N=2880 2x8, lookup-table path",
    "lut1": ("aq_linear, T=1 K=8192 N=65536 2x8 (134 MB of codes, more than L2), AUTO: the "
             "rotated-table kernel (bank-conflict-free tables, one fp32 per entry)"),
    "book16_decode": "aq_decode of the 2^16-codebook conv weight (960 x 8640, 1x16)",
    "book16_gemm": ("aq_conv2d_nhwc 2x8x8x960->960 1x16, weights decoded beforehand (the "
                    "tensor-core GEMM alone)"),
    "grad": "aq_codebook_grad of the qkv layer (fp32 G)",
    "search": "aq_code_update of the qkv layer, both codebooks, unweighted",
}


def run_kernel_workload(args, aq, torch, dev, stream):
    """One kernel's call on the seeded qkv-shaped layer, --warmup + --steps plain launches
    (no graph), for ncu captures; returns the mean time per call (CUDA events)."""
    from aq_synth import SEEDS, WORKLOADS, LinearSpec, make_conv, make_linear
    w = args.workload
    if w.startswith("book16"):
        L = Dev(aq, torch, make_conv(WORKLOADS["conv8_book16"], seed=SEEDS["conv8_book16"]), dev,
                path=aq.AQ_PATH_PREDECODED)
        L.quant(stream)
        if w == "book16_decode":
            wdec = torch.empty((L.N, L.K), dtype=torch.float16, device=dev)
            call = lambda: L.decode_only(stream, wdec)
        else:
            L.decode_only(stream, L.ws)
            call = lambda: L.layer(stream)
    elif w in ("fused128", "few4", "lut8", "lut1"):
        T = {"fused128": 128, "few4": 4, "lut8": 8, "lut1": 1}[w]
        K, N = (8192, 65536) if w == "lut1" else (960, 2880)
        spec = LinearSpec(T=T, K=K, N=N, M=2, B=8, cb_std=0.05, act="uniform", s_x=0.02)
        L = Dev(aq, torch, make_linear(spec, seed=7), dev, path=3 if w == "lut8" else 0)
        call = lambda: L.layer(stream)
    else:
        L = Dev(aq, torch, make_linear(WORKLOADS["qkv"], seed=SEEDS["qkv"]), dev)
        N, K = L.N, L.K
        if w == "quant":
            call = lambda: L.quant(stream)
        elif w == "decode":
            wdec = torch.empty((N, K), dtype=torch.float16, device=dev)
            call = lambda: L.decode_only(stream, wdec)
        elif w == "linear_f16":
            call = lambda: L.step_f16(stream)
        elif w == "gemm_a16":
            L.quant(stream)
            xh = L.xq.to(torch.float16)
            wsp = torch.empty(aq.aq_linear_a16_workspace_size(L.T, K, N, 8, L.M, L.B,
                                                              aq.AQ_PATH_PREDECODED),
                              dtype=torch.uint8, device=dev)
            L.decode_only(stream, wsp)
            call = lambda: L.gemm_a16(stream, xh, wsp)
        elif w == "grad":
            G = torch.randn((N, K), dtype=torch.float32, device=dev,
                            generator=torch.Generator(device=dev).manual_seed(0))
            dC = torch.zeros((2, 256, 8), dtype=torch.float32, device=dev)
            call = lambda: aq.aq_codebook_grad(L.packed, G, L.scale, L.s_x, dC, N, K, 8, 2, 8,
                                               stream=stream)
        else:
            Wt = torch.randn((N, K), dtype=torch.float32, device=dev,
                             generator=torch.Generator(device=dev).manual_seed(0)) * 0.05
            codes = torch.randint(0, 256, (N, K // 8, 2), dtype=torch.uint8, device=dev,
                                  generator=torch.Generator(device=dev).manual_seed(1))
            call = lambda: aq.aq_code_update(Wt, L.books, codes, None, 0, 2, N, K, 8, 2, 8,
                                             stream=stream)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            call()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            call()
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / max(1, args.steps)


def small_t_sweep(aq, torch, dev, stream, reps=50):
    """Layer time against the token count T in {1, 2, 4, ..., 64} on the attention-projection
    shape (K=960, N=2880, 2x8) and on the 2^16-codebook conv's GEMM shape taken as a linear
    layer (K=8640, N=960, 1x16), on every path that runs the shape.  Per path: the step
    (quantizer + layer, fp16 output) with warm L2 (a graph of 8 launches replayed) and cold L2
    (a 256 MB buffer written before each launch: a graph of 8 x (write, step) minus a graph of
    the 8 writes).  The roofline is
    max(flops / tensor peak, algorithmic bytes / HBM bandwidth), the bytes being codes,
    codebooks, int8 activations, fp16 output, scale and bias."""
    from aq_synth import LinearSpec, make_linear
    peaks = measured_peaks()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    names = {aq.AQ_PATH_AUTO: "auto", aq.AQ_PATH_DENSE: "dense", aq.AQ_PATH_FUSED: "fused",
             aq.AQ_PATH_LUT: "lut", aq.AQ_PATH_FEW_TOKENS: "few"}
    rows = []
    for shape, K, N, M, B in (("attention qkv K=960 N=2880 2x8", 960, 2880, 2, 8),
                              ("2^16-codebook K=8640 N=960 1x16", 8640, 960, 1, 16)):
        for T in (1, 2, 4, 8, 16, 32, 64):
            spec = LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05, act="uniform", s_x=0.02)
            inp = make_linear(spec, seed=11 + T)
            fl = 2.0 * T * N * K
            by = N * K * M * B // 64 + M * (1 << B) * 16 + T * K + 2 * T * N + 4 * N
            roof = max(fl / (peaks["bf16_tflops"] * 1e12), by / (peaks["hbm_gbs"] * 1e9)) * 1e6
            row = {"shape": shape, "T": T, "roofline_us": round(roof, 3),
                   "bound": "hbm" if by / peaks["hbm_gbs"] > fl / (peaks["bf16_tflops"] * 1e3)
                   else "tensor",
                   "auto_path": names[aq.aq_linear_plan(T, K, N, 8, M, B, 0)["path"]]}
            for path, pname in names.items():
                try:
                    aq.aq_linear_plan(T, K, N, 8, M, B, path)
                except aq.AQError:
                    continue
                L = Dev(aq, torch, inp, dev, path=path)
                with torch.cuda.stream(stream):
                    for _ in range(3):
                        L.step(stream)
                stream.synchronize()
                g = capture(torch, stream, lambda: [L.step(stream) for _ in range(8)])
                warm = replay_ms(torch, stream, g, reps) / 8 * 1e3
                # cold: 8 x (flush, step) minus 8 x flush, both graphs replayed
                gc = capture(torch, stream, lambda: [(flush.fill_(1), L.step(stream))
                                                     for _ in range(8)])
                gf = capture(torch, stream, lambda: [flush.fill_(1) for _ in range(8)])
                cold = (replay_ms(torch, stream, gc, 10) - replay_ms(torch, stream, gf, 10)) / 8
                del g, gc, gf
                assert aq.aq_device_error() == 0
                row[pname] = {"warm_us": round(warm, 2), "cold_us": round(cold * 1e3, 2)}
                del L
            rows.append(row)
            print(json.dumps(row), flush=True)
    return rows


def run_single(args):
    """One non-headline workload on one GPU (profiling aid): prints its timing."""
    import torch
    import paper_2506_05960_gb300 as aq
    from aq_synth import SEEDS, WORKLOADS, make_conv
    dev = torch.device("cuda", 0)
    aq.load_library()
    stream = torch.cuda.Stream(device=dev)
    if args.workload in KERNEL_WORKLOADS:
        ms = run_kernel_workload(args, aq, torch, dev, stream)
        out = {"workload": KERNEL_WORKLOADS[args.workload], "us_per_call": ms * 1e3,
               "timing": "plain launches, CUDA events (no graph)"}
    elif args.workload == "tsweep":
        small_t_sweep(aq, torch, dev, stream)
        return 0
    elif args.workload == "unet":
        ms, gflop, nl = unet_forward(aq, torch, dev, stream, 2, reps=max(1, args.steps // 100))
        out = {"workload": "UNet-shaped forward W2A8 batch 2", "ms_per_forward": ms,
               "gflop": gflop, "layers": nl}
    else:
        name = "conv64" if args.workload == "conv64" else "conv8_book16"
        L = Dev(aq, torch, make_conv(WORKLOADS[name], seed=SEEDS[name]), dev)
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                L.step(stream)
        stream.synchronize()
        gl = capture(torch, stream, lambda: [L.step(stream) for _ in range(8)])
        ms = replay_ms(torch, stream, gl, max(1, args.steps // 8)) / 8
        out = {"workload": args.workload, "us_per_step": ms * 1e3,
               "tflops": L.flops / (ms * 1e-3) / 1e12}
    assert aq.aq_device_error() == 0
    print(json.dumps(out), flush=True)
    return 0


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=100)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the other workloads and the UNet-shaped forward")
    ap.add_argument("--unet-batches", default="2,16,64",
                    help="batches of the UNet-shaped forward extras (comma separated)")
    ap.add_argument("--cpu-oracle", choices=["single", "all"], default=None,
                    help=argparse.SUPPRESS)   # child process of the CPU baselines
    ap.add_argument("--no-cpu-baselines", action="store_true",
                    help="skip the per-workload CPU oracle timings")
    ap.add_argument("--workload", default="qkv",
                    choices=["qkv", "conv64", "conv8", "unet", "tsweep"] + list(KERNEL_WORKLOADS),
                    help="qkv: the headline line (default); the others run only that workload "
                         "and print its timing (for profiling)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    if args.cpu_oracle:
        cpu_oracle_child(args.cpu_oracle, min(args.cpu_seconds, 2.0))
        return 0
    if args.impl == "reference":
        return run_reference(args)
    if args.workload != "qkv":
        return run_single(args)

    world, rank, local = dist_setup()
    spec, sets = headline_sets(NSETS)
    T, K, N, g, M, B = spec.T, spec.K, spec.N, spec.g, spec.M, spec.B
    fl = linear_flops(T, N, K)

    # CPU baseline first (before any GPU work), rank 0 at N=1 only
    cpu = None
    cpu_all = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = time_oracle(sets[0], fl, min_seconds=args.cpu_seconds)
        if not args.no_cpu_baselines and not args.no_extras:
            cpu_all = run_cpu_baselines()

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

    bufs = [Dev(aq, torch, inp, dev) for inp in sets]
    wdec = torch.empty((N, K), dtype=torch.float16, device=dev)
    torch.cuda.synchronize()
    stream = torch.cuda.Stream(device=dev)

    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            bufs[i % NSETS].step_f16(stream)
            bufs[i % NSETS].step(stream)
    stream.synchronize()
    assert aq.aq_device_error() == 0

    # graphs: the step over the 8 buffer sets, and over the first (steps % 8) of them, so
    # that exactly --steps steps are timed
    full_reps, rem = divmod(max(1, args.steps), NSETS)
    g_main = capture(torch, stream, lambda: [b.step_f16(stream) for b in bufs]) if full_reps else None
    g_rem = capture(torch, stream, lambda: [b.step_f16(stream) for b in bufs[:rem]]) if rem else None
    for gg in (g_main, g_rem):
        if gg is not None:
            gg.replay()
    stream.synchronize()

    steps = full_reps * NSETS + rem
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    sampler = ClockSampler(local)
    sampler.start()
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        ev[0].record(stream)
        for _ in range(full_reps):
            g_main.replay()
        if g_rem is not None:
            g_rem.replay()
        ev[1].record(stream)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    ms_total = ev[0].elapsed_time(ev[1])
    assert aq.aq_device_error() == 0
    if pg:
        ms_total = max_over_ranks(pg, ms_total, dev)
    ms_step = ms_total / steps
    value = job_throughput(world, fl, ms_step)

    # the dominant kernel by itself: a graph of 8 GEMM launches (one per buffer set, fp16
    # activation codes, weights decoded beforehand), replayed >= 50 times and >= 20 ms; and
    # the decode alone the same way
    for b in bufs:
        b.quant(stream)
    xh = [b.xq.to(torch.float16) for b in bufs]
    ws_pre = [torch.empty(aq.aq_linear_a16_workspace_size(T, K, N, g, M, B, aq.AQ_PATH_PREDECODED),
                          dtype=torch.uint8, device=dev) for _ in bufs]
    for b, w in zip(bufs, ws_pre):
        b.decode_only(stream, w)
    stream.synchronize()
    g_gemm = capture(torch, stream, lambda: [b.gemm_a16(stream, x, w)
                                             for b, x, w in zip(bufs, xh, ws_pre)])
    g_decode = capture(torch, stream, lambda: [b.decode_only(stream, wdec) for b in bufs])

    def per_launch_us(gg):
        est = replay_ms(torch, stream, gg, 5)
        reps = max(50, int(20.0 / max(est, 1e-3)) + 1)
        return replay_ms(torch, stream, gg, reps) / NSETS * 1e3, reps

    gemm_us, gemm_reps = per_launch_us(g_gemm)
    decode_us, _ = per_launch_us(g_decode)
    clocks = sampler.stop()
    assert aq.aq_device_error() == 0
    gemm_ms = gemm_us * 1e-3
    gemm_plan = aq.aq_linear_f16_plan(T, K, N, g, M, B, aq.AQ_PATH_AUTO)
    # cross-check: the library's CUDA event pairs around each kernel over plain launches of the
    # step (an event between two kernels also waits out the programmatic-launch overlap, so a
    # pair includes the kernel's set-up: an upper bound)
    aq.aq_profile_enable(True)
    with torch.cuda.stream(stream):
        for i in range(64):
            bufs[i % NSETS].step_f16(stream)
    stream.synchronize()
    prof = aq.aq_profile_read()
    aq.aq_profile_enable(False)
    prof_us = {k: (v[0] / v[1] * 1e3 if v[1] else None) for k, v in prof.items() if v[1]}
    del g_gemm, g_decode, ws_pre, xh

    peaks = measured_peaks()
    achieved = fl / (gemm_ms * 1e-3) / 1e12
    traffic = TRAFFIC["bytes"] if TRAFFIC.get("sources_sha") == sources_sha() else None
    launches_per_step = 3    # quantizer, decode, GEMM (the headline plan does not split K)

    # e2e through the public API: every step copies its fp16 input from pinned host memory,
    # runs aq_linear_f16 and copies its fp16 output back to pinned host memory.
    #  - serial: copy in, step, copy out on one stream (each step waits for its copies);
    #  - pipelined (the reported e2e): the serving pattern -- copy-in, compute and copy-out
    #    streams with two buffer slots, so step i's compute overlaps the input copy of step
    #    i+1 and the output copy of step i-1 on the two copy engines.  Every step still
    #    moves all of its bytes between host and device inside the timed region.
    h_x = [b.x16.cpu().pin_memory() for b in bufs[:2]]
    h_y = [torch.empty((T, N), dtype=torch.float16).pin_memory() for _ in range(2)]
    e2e_steps = max(1, args.e2e_steps)

    def e2e_serial(n):
        for i in range(n):
            b = bufs[i % 2]
            b.x16.copy_(h_x[i % 2], non_blocking=True)
            b.step_f16(stream)
            h_y[i % 2].copy_(b.y, non_blocking=True)

    s_in = torch.cuda.Stream(device=dev)
    s_out = torch.cuda.Stream(device=dev)

    def e2e_pipelined(n):
        ev_in = [torch.cuda.Event() for _ in range(2)]     # input slot filled
        ev_cmp = [torch.cuda.Event() for _ in range(2)]    # step done (input read, y written)
        ev_out = [torch.cuda.Event() for _ in range(2)]    # output slot copied out
        for i in range(n):
            k = i % 2
            b = bufs[k]
            with torch.cuda.stream(s_in):
                if i >= 2:
                    s_in.wait_event(ev_cmp[k])              # the step that read x16[k] is done
                b.x16.copy_(h_x[k], non_blocking=True)
                ev_in[k].record(s_in)
            stream.wait_event(ev_in[k])
            if i >= 2:
                stream.wait_event(ev_out[k])                # y[k] of step i-2 copied out
            with torch.cuda.stream(stream):
                b.step_f16(stream)
                ev_cmp[k].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_cmp[k])
                h_y[k].copy_(b.y, non_blocking=True)
                ev_out[k].record(s_out)

    def time_e2e(fn):
        # the compute stream is torch's current stream here, so copies that name no stream
        # (the serial variant) are ordered with the steps on it
        with torch.cuda.stream(stream):
            fn(4)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            s_in.wait_stream(stream)
            s_out.wait_stream(stream)
            fn(e2e_steps)
            stream.wait_stream(s_in)
            stream.wait_stream(s_out)
            e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / e2e_steps
        if pg:
            ms = max_over_ranks(pg, ms, dev)
        return ms

    def copies_only(n):
        # the same host <-> device copies with no compute: the floor of the pipelined loop
        for i in range(n):
            k = i % 2
            with torch.cuda.stream(s_in):
                bufs[k].x16.copy_(h_x[k], non_blocking=True)
            with torch.cuda.stream(s_out):
                h_y[k].copy_(bufs[k].y, non_blocking=True)

    e2e_serial_ms = time_e2e(e2e_serial)
    e2e_ms = time_e2e(e2e_pipelined)
    # every step's output reached the host: the last two slots hold the last two steps
    y_last = bufs[(e2e_steps - 1) % 2].y.cpu()
    assert torch.equal(h_y[(e2e_steps - 1) % 2], y_last)
    copy_ms = time_e2e(copies_only)

    # the other workloads (per layer, graph replay) and the UNet-shaped forward
    layers, unet = {}, None
    if not args.no_extras and rank == 0:
        # context, not the product path: a library fp16 GEMM (cuBLAS through torch.mm) of the
        # same contraction shapes on fp16 operands already in HBM -- no int8 operand, no
        # weight decode, no scale/bias epilogue -- 8 rotating buffer sets, CUDA graph replay
        lib = {}
        for name, (Tm, Km, Nm) in (("qkv T=4096 K=960 N=2880", (T, K, N)),
                                   ("conv 16x64x64x192->192 as a GEMM T=65536 K=1728 N=192",
                                    (65536, 1728, 192))):
            gen = torch.Generator(device=dev).manual_seed(7)
            As = [torch.randn((Tm, Km), dtype=torch.float16, device=dev, generator=gen)
                  for _ in range(NSETS)]
            Ws = [torch.randn((Nm, Km), dtype=torch.float16, device=dev, generator=gen)
                  for _ in range(NSETS)]
            Ys = [torch.empty((Tm, Nm), dtype=torch.float16, device=dev) for _ in range(NSETS)]

            def mm():
                for a, w, y in zip(As, Ws, Ys):
                    torch.mm(a, w.t(), out=y)
            with torch.cuda.stream(stream):
                for _ in range(3):
                    mm()
            stream.synchronize()
            gm = capture(torch, stream, mm)
            ms = replay_ms(torch, stream, gm, 20) / NSETS
            tf = linear_flops(Tm, Nm, Km) / (ms * 1e-3) / 1e12
            lib[name] = {"us_per_gemm": ms * 1e3, "tflops": tf,
                         "tensor_roofline_frac": tf / peaks["bf16_tflops"]}
            del gm, As, Ws, Ys
        lib["what"] = ("cuBLAS fp16 GEMM (torch.mm, fp32 accumulate) of the same shape on fp16 "
                       "operands, no decode/int8 conversion/epilogue; context for the GEMM's "
                       "roofline fraction at this shape")
        lib["aq_gemm_over_cublas_qkv"] = achieved / lib["qkv T=4096 K=960 N=2880"]["tflops"]
        layers["library GEMM of the same shapes (context)"] = lib
        torch.cuda.empty_cache()
        # the fixed cost of one dependent launch under graph replay: our quantizer on 16
        # elements (the least work a library kernel can do), 8 launches per graph
        fx = torch.zeros(16, dtype=torch.float16, device=dev)
        fq = torch.empty(16, dtype=torch.int8, device=dev)
        gfl = capture(torch, stream, lambda: [aq.aq_quant_act(fx, fq, 16, 0.02, stream=stream)
                                              for _ in range(8)])
        floor_us = replay_ms(torch, stream, gfl, 50) / 8 * 1e3
        del gfl
        layers["launch floor (one dependent library launch, graph replay)"] = {
            "us_per_launch": floor_us,
            "what": "aq_quant_act on 16 elements, 8 launches per CUDA graph: the per-launch "
                    "fixed cost that bounds the token-poor layers below"}
        from aq_synth import SEEDS, WORKLOADS, make_conv
        for name, wl in (("conv3x3 16x64x64x192->192 W4A8 (4x8)", "conv64"),
                         ("conv3x3 2x8x8x960->960 one 2^16 codebook (1x16)", "conv8_book16")):
            L = Dev(aq, torch, make_conv(WORKLOADS[wl], seed=SEEDS[wl]), dev)
            with torch.cuda.stream(stream):
                for _ in range(3):
                    L.step(stream)
            stream.synchronize()
            gl = capture(torch, stream, lambda: [L.step(stream) for _ in range(8)])
            ms = replay_ms(torch, stream, gl, 20) / 8
            s_ = L.spec
            plan = aq.aq_conv2d_plan(s_.Nb, s_.H, s_.W, s_.Cin, s_.Cout, 3, 3, s_.stride, 1, 8,
                                     L.M, L.B, L.path)
            layers[name] = {"us_per_step": ms * 1e3,
                            "tflops": L.flops / (ms * 1e-3) / 1e12,
                            "tensor_roofline_frac": L.flops / (peaks["bf16_tflops"] * 1e12) / (ms * 1e-3),
                            "plan": plan,
                            "launch_floor_us": floor_us,
                            "step": "quantizer + layer (AUTO path), CUDA graph replay"}
            del gl, L
        # backward of Eq. 4 (codebook gradient) on the headline layer: HBM-bound read of G
        gsets = []
        for i in range(NSETS):
            gsets.append(torch.randn((N, K), dtype=torch.float32, device=dev,
                                     generator=torch.Generator(device=dev).manual_seed(i)))
        dC = torch.zeros((M, 1 << B, g), dtype=torch.float32, device=dev)
        gb = bufs[0]

        def cgrad():
            for G in gsets:
                aq.aq_codebook_grad(gb.packed, G, gb.scale, gb.s_x, dC, N, K, g, M, B,
                                    stream=stream)
        with torch.cuda.stream(stream):
            cgrad()
        stream.synchronize()
        gc = capture(torch, stream, cgrad)
        ms = replay_ms(torch, stream, gc, 20) / NSETS
        cg_bytes = N * K * 4 + aq.aq_packed_size(N, K, g, M, B) + 2 * N + M * (1 << B) * g * 4
        layers["codebook gradient of the qkv layer (fp32 G, 2x8)"] = {
            "us_per_step": ms * 1e3, "gbs": cg_bytes / (ms * 1e-3) / 1e9,
            "hbm_roofline_frac": cg_bytes / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "bytes_per_call": cg_bytes,
            "step": "aq_codebook_grad, 8 rotating G buffers (> L2), CUDA graph replay"}
        del gc, gsets
        # input gradient of the qkv layer (dL/dX = dY diag(scale) W-hat: transposed decode +
        # the fp16-activation GEMM over N), 8 rotating dY buffers
        dys = [torch.randn((T, N), device=dev, generator=torch.Generator(device=dev).manual_seed(
            20 + i)).to(torch.float16) for i in range(NSETS)]
        dxs = [torch.empty((T, K), dtype=torch.float16, device=dev) for _ in range(NSETS)]
        igb = aq.aq_linear_input_grad_workspace_size(T, K, N, g, M, B)
        igws = [torch.empty(igb, dtype=torch.uint8, device=dev) for _ in range(NSETS)]

        def igrad():
            for dy_, dx_, w_ in zip(dys, dxs, igws):
                aq.aq_linear_input_grad(dy_, 1.0, gb.packed, gb.books, gb.scale, dx_,
                                        aq.AQ_DTYPE_F16, T, K, N, g, M, B, w_, igb, stream=stream)
        with torch.cuda.stream(stream):
            igrad()
        stream.synchronize()
        gi = capture(torch, stream, igrad)
        ms = replay_ms(torch, stream, gi, 20) / NSETS
        layers["input gradient of the qkv layer (dL/dX, fp16 dY, 2x8)"] = {
            "us_per_step": ms * 1e3, "tflops": fl / (ms * 1e-3) / 1e12,
            "tensor_roofline_frac": fl / (ms * 1e-3) / 1e12 / peaks["bf16_tflops"],
            "step": ("aq_linear_input_grad (transposed scaled decode + tensor-core GEMM over N), "
                     "8 rotating dY buffers, CUDA graph replay")}
        del gi, dys, dxs, igws
        # Stage-1 code search (one greedy step over both codebooks) on the qkv layer
        from aq_synth import make_linear as _ml
        inp1 = _ml(WORKLOADS["qkv"], seed=SEEDS["qkv"])
        Wt = torch.from_numpy(np.ascontiguousarray(
            (inp1["codebooks"].astype(np.float32)[0][inp1["codes"][:, :, 0]]
             + inp1["codebooks"].astype(np.float32)[1][inp1["codes"][:, :, 1]]).reshape(N, K)
            + np.float32(0.01))).to(dev)
        books_cs = torch.from_numpy(inp1["codebooks"]).to(dev)
        codes_cs = torch.from_numpy(np.ascontiguousarray(inp1["codes"])).to(dev)
        Hb = torch.eye(8, device=dev).expand(K // 8, 8, 8).contiguous()
        for weighted in (False, True):
            def cs():
                aq.aq_code_update(Wt, books_cs, codes_cs, Hb if weighted else None, 0, M, N, K,
                                  8, M, 8, stream=stream)
            with torch.cuda.stream(stream):
                cs()
            stream.synchronize()
            gcs = capture(torch, stream, cs)
            ms = replay_ms(torch, stream, gcs, 10)
            cand = N * (K // 8) * M * 256
            layers["code search step of the qkv layer (2x8, " + ("H-weighted" if weighted
                                                                 else "unweighted") + ")"] = {
                "us_per_step": ms * 1e3, "candidates_per_s": cand / (ms * 1e-3),
                "step": "aq_code_update over both codebooks, CUDA graph replay"}
            del gcs
        # small-T sweep on the qkv shape (2x8) and the 2^16-codebook shape (K = 8640, N = 960,
        # 1x16): per path, to locate where the lookup-table, fused and dense orders cross
        from aq_synth import LinearSpec, make_linear as _mlin
        sweep = {}
        for (Ks, Ns, Ms, Bs, paths) in ((960, 2880, 2, 8, (0, 1, 2, 3)), (8640, 960, 1, 16, (0, 1, 2))):
            for Ts in (1, 2, 4, 8, 16, 32, 64):
                inp_s = _mlin(LinearSpec(T=Ts, K=Ks, N=Ns, M=Ms, B=Bs), seed=Ts)
                for pth in paths:
                    if pth == 3 and Ts > 16:
                        continue
                    Ls = [Dev(aq, torch, inp_s, dev, path=pth) for _ in range(NSETS)]
                    with torch.cuda.stream(stream):
                        for L in Ls:
                            L.step(stream)
                    stream.synchronize()
                    gs = capture(torch, stream, lambda: [L.step(stream) for L in Ls])
                    ms = replay_ms(torch, stream, gs, 20) / NSETS
                    wbytes = alg_bytes(Ts, Ks, Ns, Ms, Bs)
                    key = f"K={Ks} N={Ns} {Ms}x{Bs} T={Ts} " + ["AUTO", "DENSE", "FUSED", "LUT"][pth]
                    sweep[key] = {"us_per_step": ms * 1e3,
                                  "tflops": Ls[0].flops / (ms * 1e-3) / 1e12,
                                  "hbm_gbs_algorithmic": wbytes / (ms * 1e-3) / 1e9,
                                  "hbm_roofline_frac": wbytes / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"]}
                    del gs, Ls
        # few tokens on a layer large enough to amortise the launches: how fast each path
        # streams the codes (K=8192, N=16384, 2x8: 33.6 MB of codes; N=65536: 134 MB, more
        # than L2); AUTO takes the table path up to four tokens here
        for Ts, Ns, pth in ((1, 16384, aq.AQ_PATH_FEW_TOKENS), (1, 16384, aq.AQ_PATH_AUTO),
                            (2, 16384, aq.AQ_PATH_FEW_TOKENS), (2, 16384, aq.AQ_PATH_AUTO),
                            (4, 16384, aq.AQ_PATH_FEW_TOKENS), (4, 16384, aq.AQ_PATH_FUSED),
                            (4, 16384, aq.AQ_PATH_AUTO), (1, 65536, aq.AQ_PATH_AUTO)):
            inp_s = _mlin(LinearSpec(T=Ts, K=8192, N=Ns, M=2, B=8), seed=90 + Ts)
            Ls = [Dev(aq, torch, inp_s, dev, path=pth) for _ in range(4)]
            with torch.cuda.stream(stream):
                for L in Ls:
                    L.step(stream)
            stream.synchronize()
            gs = capture(torch, stream, lambda: [L.layer(stream) for L in Ls])
            ms = replay_ms(torch, stream, gs, 10) / len(Ls)
            wbytes = alg_bytes(Ts, 8192, Ns, 2, 8)
            pname = {aq.AQ_PATH_FEW_TOKENS: "FEW", aq.AQ_PATH_AUTO: "AUTO (table)",
                     aq.AQ_PATH_FUSED: "FUSED"}[pth]
            sweep[f"K=8192 N={Ns} 2x8 T={Ts} {pname} (layer only, 4 rotating buffer sets)"] = {
                "us_per_step": ms * 1e3, "hbm_gbs_algorithmic": wbytes / (ms * 1e-3) / 1e9,
                "hbm_roofline_frac": wbytes / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"]}
            del gs, Ls
            torch.cuda.empty_cache()
        layers["small-T sweep (quantizer + layer per step, 8 rotating buffer sets)"] = sweep
        unet = {}
        for Mu, label in ((2, "W2A8"), (4, "W4A8")):
            for batch in [int(b) for b in args.unet_batches.split(",") if b]:
                for fq, ahead, mixed in ((False, False, False), (True, False, False),
                                         (True, True, False), (True, True, True)):
                    ms, gflop, nl = unet_forward(aq, torch, dev, stream, Mu, batch=batch,
                                                 reps=20 if batch <= 2 else 5, fused_quant=fq,
                                                 decode_ahead=ahead, mixed=mixed)
                    key = (f"{label} batch {batch}" + (" quantizer in epilogue" if fq else "")
                           + (", decode ahead" if ahead else "")
                           + (", fp16 codes into the layers whose plan prefers them"
                              if mixed else ""))
                    unet[key] = {"ms_per_forward": ms, "gflop": gflop, "tflops": gflop / ms,
                                 "layers": nl, "batch": batch,
                                 "step": ("each layer writes the next layer's activation codes "
                                          "(int8, or fp16 values where that layer's plan reads "
                                          "them faster)" if mixed else
                                          "each layer writes the next layer's int8 activations"
                                          if fq else "each layer preceded by aq_quant_act")
                                         + ("; dense-path layers decoded on a second stream "
                                            "ahead of the chain (AQ_PATH_PREDECODED)"
                                            if ahead else "")}
                    torch.cuda.empty_cache()
        assert aq.aq_device_error() == 0

    step_frac = (max(fl / (peaks["bf16_tflops"] * 1e12),
                     alg_bytes(T, K, N, M, B) / (peaks["hbm_gbs"] * 1e9)) / (ms_step * 1e-3))
    if rank == 0:
        line = {
            "metric": METRIC,
            "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
            "config": {"workload": HEADLINE, "T": T, "K": K, "N": N, "g": g, "M": M, "B": B,
                       "parallelism": f"replicas{world}",
                       "l2": f"inputs larger than L2: {NSETS} rotating buffer sets",
                       "timing": (f"exactly {steps} steps: {full_reps} CUDA graph replay(s) of "
                                  f"{NSETS} steps + one graph of {rem} step(s), CUDA events")},
            "hbm_gbs_algorithmic": alg_bytes(T, K, N, M, B) / (ms_step * 1e-3) / 1e9,
            "roofline": {"bound": "tensor", "kernel": "aq_gemm_kernel", "achieved": achieved,
                         "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": achieved / peaks["bf16_tflops"], "traffic": traffic,
                         "peak_source": f"{peaks['source']} bf16 dense burst (the fp16 rate is equal)",
                         "frac_of_sustained": (achieved / peaks["bf16_tflops_sustained"]
                                               if peaks.get("bf16_tflops_sustained") else None),
                         "kernel_us": gemm_us,
                         "kernel_timing": (f"graph of {NSETS} GEMM launches (one per buffer set, "
                                           f"weights decoded beforehand) replayed {gemm_reps} "
                                           "times, CUDA events"),
                         "kernel_plan": gemm_plan,
                         "kernel_us_event_pairs": prof_us.get("gemm"),
                         "step_frac": step_frac},
            "step_us": {"total": ms_step * 1e3, "gemm": gemm_us, "decode": decode_us,
                        "quantizer_and_gaps": ms_step * 1e3 - gemm_us - decode_us,
                        "event_pairs_plain_launches": prof_us},
            "step_roofline_frac": step_frac,
            "cpu_baseline": cpu,
            "e2e": {"value": job_throughput(world, fl, e2e_ms), "unit": "TFLOP/s",
                    "ms_per_step": e2e_ms, "h2d_bytes_per_step": T * K * 2,
                    "d2h_bytes_per_step": T * N * 2,
                    "how": ("aq_linear_f16 from pinned host input to pinned host output, copy-in / "
                            "compute / copy-out streams overlapped across consecutive steps"),
                    "copy_floor_ms_per_step": copy_ms,
                    "copy_floor_how": ("the step's input and output copies alone, on the "
                                       "copy-in and copy-out streams (no compute)"),
                    "serial": {"value": job_throughput(world, fl, e2e_serial_ms),
                               "ms_per_step": e2e_serial_ms,
                               "how": "copy in, step, copy out on one stream"}},
            "gpu_launches": launches_per_step * steps,
            "clocks": clocks,
        }
        if cpu_all:
            line["cpu_baselines"] = cpu_all
        if layers:
            line["layers"] = layers
        if unet:
            line["unet_forward"] = unet
        print(json.dumps(line), flush=True)
    if pg:
        pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
