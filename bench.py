#!/usr/bin/env python
"""Decode throughput of the Llama-2-7B sparse linear stack on GB300.

A step is one decode step through the linear layers of all 32 Llama-2-7B layers:
per layer the fused qkv (4096->12288), o (4096->4096), fused gate/up (4096->22016)
and down (11008->4096) projections, 70% unstructured per-row magnitude sparsity,
bf16 weights in the bitmask-compressed format, x bf16 [M, K], FP32 accumulation,
bf16 y.  tok/s = M / step time.  The 32 layers are 32 distinct device copies of one
seeded layer, so every step streams 4.7 GB (> L2) of compressed weights from HBM.
Further sections: the same step with its elementwise glue (residual adds, gate*up) as one
persistent sp_chain_run launch and as a CUDA graph of separate launches; the INT8 stack;
prefill.

  python bench.py [--gpus N --steps K --warmup W --m M]        our CUDA path
  python bench.py --impl reference ...                          the float64 CPU oracle

One compact JSON line on stdout (rank 0, about 2 KB: the headline figures, the roofline of
the dominant kernel, the CPU baseline, clocks and a summary of the context sections; the
sections in full go to --sections-out).  With --gpus N > 1 (under torchrun) every rank
runs an independent replica (weak scaling; no collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Llama-2-7B sparse-linear decode tok/s @70%; achieved HBM GB/s vs roofline"
SHAPES = ["qkv", "o", "gate_up", "down"]
LAYERS = 32


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--m", type=int, default=1, help="decode batch (tokens per step)")
    ap.add_argument("--pct", type=int, default=70)
    ap.add_argument("--path", default="auto", choices=["auto", "cuda_core", "tensor_core"])
    ap.add_argument("--sweep", default="1,4,16", help="extra batch sizes reported under per_m ('' = none)")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle leg")
    ap.add_argument("--no-stack", action="store_true", help="skip the INT8 32-layer stack section")
    ap.add_argument("--no-chain", action="store_true", help="skip the chained-step (glue included) section")
    ap.add_argument("--layers", type=int, default=32, help="profiling aid (--single chain): layers in the chain")
    ap.add_argument("--int8", action="store_true", help="profiling aid (--single <shape>): INT8 values + fp32 scales")
    ap.add_argument("--update", action="store_true",
                    help="with --single <shape>: time the masked weight update (sp_masked_update) instead of the linear")
    ap.add_argument("--no-prefill", action="store_true", help="skip the M=2048 prefill section")
    ap.add_argument("--no-dense", action="store_true", help="skip the dense cuBLAS comparison section")
    ap.add_argument("--no-update", action="store_true", help="skip the masked weight update section")
    ap.add_argument("--no-w8a8", action="store_true", help="skip the INT8-activation (W8A8) section")
    ap.add_argument("--square-sweep", action="store_true",
                    help="run only the 12288 x 12288 sparse matmul at 0-90%% sparsity (M = 2048, tensor cores)")
    ap.add_argument("--no-square", action="store_true", help="skip the 12288 x 12288 sparsity sweep section")
    ap.add_argument("--no-profile", action="store_true", help="skip the per-layer sparsity profile section")
    ap.add_argument("--no-sweep-config", action="store_true",
                    help="skip the sparsity x batch sweep (gate_up/down, non-uniform masks, M = 1..256)")
    ap.add_argument("--sections-out", default="",
                    help="write the full context sections (per-M tables, chained step, INT8 stack, prefill, dense "
                         "comparison, masked update, sweep) to this JSON file; the stdout line carries a summary")
    ap.add_argument("--single", default="", choices=["", "chain", *SHAPES],
                    help="profiling aid: time one layer-0 linear of this shape, or the chained step of --layers "
                         "layers (--warmup then --steps launches)")
    return ap.parse_args()


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), int(os.environ.get("WORLD_SIZE", 1))


def host_layer(pct: int, M: int):
    """Seeded host inputs of layer 0: W, mask and x per shape (the oracle's inputs)."""
    from paper_2405_03594_gb300 import synth

    out = {}
    for name in SHAPES:
        W, mask, x = synth.layer_inputs(name, pct, M, seed=0, layer=0)
        out[name] = (W, mask, x)
    return out


def algorithmic_bytes(info, M: int, K: int, N: int) -> int:
    """Compressed-weight bytes the method must read (values + one bit per weight,
    plus INT8 scales) plus the activations read and the outputs written."""
    esize = 1 if info.dtype == 1 else 2
    return int(info.nnz) * esize + N * K // 8 + int(info.scale_bytes) + 2 * M * K + 2 * M * N


def max_over_ranks(vals, device=None):
    """Element-wise maximum of `vals` over all ranks of the process group (the slowest
    replica sets the step time); the values themselves with one process."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in vals]
    t = torch.tensor([float(v) for v in vals], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def whole_job_tok_s(world: int, M: int, step_ms: float) -> float:
    """Tokens per second of all replicas together: every rank decodes M tokens per step."""
    return world * M / (step_ms * 1e-3)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def load_tensor_peak():
    """bf16 dense tensor peak (TFLOP/s) for a kernel timed alone (burst figure)."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    return 1900.0, "fallback"


def time_graph(g, steps, warmup):
    import torch

    for _ in range(warmup):
        g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(steps):
        g.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / steps


def stack_section(args, peak_gbs, host_bf):
    """Decode step of the 32-layer linear stack, 70% INT8 weights with fp32 per-row scales,
    layers chained by residual adds: as one CUDA graph of separate launches per step (M = 1,
    16, 64) and as one chained launch per step (M = 1, 4)."""
    import torch

    from paper_2405_03594_gb300 import sp, synth
    from paper_2405_03594_gb300.stack import ChainStack, LinearStack

    host = {}
    for name, (W, mask, _) in host_bf.items():
        q, s = synth.quantize_int8(W, mask)
        host[name] = (q, mask, s)
    st = LinearStack(layers=LAYERS, pct=args.pct, int8=True, max_m=64, host=host)
    wb = st.weight_bytes()
    out = {"workload": f"llama2-7b linear stack, {LAYERS} layers, {args.pct}% INT8 weights + fp32 per-row scales, "
                       "residual chain", "weight_bytes": wb, "graph_per_m": {}, "chain_per_m": {}}
    for M in (1, 16, 64):
        x = synth.activations(M, 4096, synth.rng(0, 0, 0, synth.STREAM_X))
        st.set_input(torch.from_numpy(x.view(np.int16)).to(st.dev).view(torch.bfloat16))
        g = st.capture(M)
        steps = max(3, min(args.steps, 100))
        ms = time_graph(g, steps, max(3, args.warmup))
        sp.check()
        finite = bool(torch.isfinite(st.h[:M].float()).all().item())
        bytes_step = wb + LAYERS * 2 * M * (4096 * 4 + 12288 + 22016 + 11008)
        out["graph_per_m"][str(M)] = {"tok_s": M / (ms * 1e-3), "ms_per_step": ms,
                                      "gbs": bytes_step / (ms * 1e-3) / 1e9,
                                      "frac_of_peak": bytes_step / (ms * 1e-3) / 1e9 / peak_gbs,
                                      "launches_per_step": st.launches_per_step(M), "activations_finite": finite}
        del g
    del st
    torch.cuda.empty_cache()
    cs = ChainStack(layers=LAYERS, pct=args.pct, int8=True, max_m=4, host=host)
    for M in (1, 4):
        ms, cu = time_chain(cs, M, max(3, min(args.steps, 100)), max(3, args.warmup), 1)
        b = chain_bytes(cs, M)
        out["chain_per_m"][str(M)] = {"tok_s": M / (ms * 1e-3), "ms_per_step": ms, "chain_us": cu,
                                      "gbs": b / (cu * 1e-6) / 1e9, "frac_of_peak": b / (cu * 1e-6) / 1e9 / peak_gbs,
                                      "launches_per_step": cs.launches_per_step(M),
                                      "activations_finite": bool(torch.isfinite(cs.h[:M].float()).all().item())}
    del cs
    torch.cuda.empty_cache()
    return out


def prefill_section(args):
    """Prefill: the four shapes at 50% and 70% sparsity, x [2048, K], tensor-core path."""
    import numpy as np
    import torch

    from paper_2405_03594_gb300 import sp, synth

    peak, kind = load_tensor_peak()
    dev = torch.device("cuda", 0)
    M = 2048
    res = {"M": M, "peak_tflops": peak, "peak_kind": f"of {kind} (bf16_tflops, burst)", "shapes": {}}
    for pct in (50, 70):
        for name in SHAPES:
            W, mask, _ = synth.layer_inputs(name, pct, 1, seed=0, layer=0)
            N, K = W.shape
            x = synth.activations(M, K, synth.rng(0, 0, synth.PROJ_IDS[name], synth.STREAM_X))
            h = sp.compress(torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16),
                            torch.from_numpy(mask).to(dev))
            xd = torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)
            y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
            ws = torch.zeros(max(h.workspace_size(M), 256), dtype=torch.uint8, device=dev)
            for _ in range(3):
                h.linear(xd, out=y, workspace=ws, path="tensor_core")
            torch.cuda.synchronize()
            reps = 10
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(reps):
                h.linear(xd, out=y, workspace=ws, path="tensor_core")
            b.record()
            torch.cuda.synchronize()
            sp.check()
            us = a.elapsed_time(b) / reps * 1e3
            nz = 2.0 * M * int(h.info.nnz) / (us * 1e-6) / 1e12
            dense = 2.0 * M * N * K / (us * 1e-6) / 1e12
            res["shapes"][f"{name}@{pct}%"] = {"us": us, "tflops_nonzero": nz, "frac_nonzero": nz / peak,
                                               "tflops_dense_executed": dense, "frac_dense_executed": dense / peak}
            del h, xd, y, ws
    torch.cuda.empty_cache()
    return res


L2_BYTES = 129e6  # GB300 L2
NOMINAL_HBM_GBS = 8000.0  # the nominal HBM3e rate the decode roofline is also quoted against
# The paper's own speedups (abstract), on the hardware it names: context only.
PAPER_SPEEDUPS = {
    "gpu_sparsity_only": {"x": 1.7, "engine": "nm-vllm", "hardware": "NVIDIA A10",
                          "what": "Llama-2 7B inference, sparse vs dense"},
    "cpu_sparsity_only": {"x": 3.0, "engine": "DeepSparse", "hardware": "AWS c7a.4xlarge (CPU)",
                          "what": "Llama-2 7B inference, sparse vs dense"},
    "cpu_sparse_int8": {"x": 8.6, "engine": "DeepSparse", "hardware": "AWS c7a.4xlarge (CPU)",
                        "what": "sparse + INT8 vs FP32 dense decode"},
}


def dense_section(host, xs, results, Ms):
    """Context for the paper's sparse-vs-dense speedups: the same layer-0 weights, unpruned,
    as dense bf16 torch.matmul (cuBLAS) launches, timed like the sparse launches (a CUDA
    graph of back-to-back calls over enough distinct weight copies to exceed 3x L2) and as
    the dense decode step (the 128 launches of 32 layers in layer order, distinct weights per
    layer, one graph: step_speedup = dense step / sparse step), and a read-only stream of
    1 GiB through a torch reduction.  Not part of the timed step; any failure is reported in
    the section instead of ending the run."""
    import numpy as np
    import torch

    out = {"how": "dense bf16 torch.matmul (cuBLAS) of the unpruned layer-0 weights, CUDA graph over "
                  "copies > 3x L2, 20 replays; speedup = dense us / sparse us per launch; step_speedup = "
                  "dense 32-layer step (128 launches in layer order, 32 weight copies per shape, one graph, "
                  "10 replays) / the sparse step",
           "shapes": {}, "step_speedup": {}, "launch_sum_speedup": {}, "paper": PAPER_SPEEDUPS}
    try:
        dev = torch.device("cuda", torch.cuda.current_device())
        dense_sum = {M: 0.0 for M in Ms}
        sparse_sum = {M: 0.0 for M in Ms}
        for name in SHAPES:
            W = host[name][0]
            N, K = W.shape
            w0 = torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16)
            copies = max(2, int(-(-3 * L2_BYTES // (2 * N * K))))
            ws = [w0] + [w0.clone() for _ in range(copies - 1)]
            rec = {}
            for M in Ms:
                x = xs[name][:M]
                y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
                for w in ws:
                    torch.matmul(x, w.t(), out=y)
                torch.cuda.synchronize()
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    for w in ws:
                        torch.matmul(x, w.t(), out=y)
                for _ in range(3):
                    g.replay()
                torch.cuda.synchronize()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                reps = 20
                a.record()
                for _ in range(reps):
                    g.replay()
                b.record()
                torch.cuda.synchronize()
                us = a.elapsed_time(b) / (reps * len(ws)) * 1e3
                sparse_us = results[M]["per_shape"][name]["us_per_launch"]
                dense_bytes = 2 * N * K + 2 * M * K + 2 * M * N
                rec[str(M)] = {"dense_us": round(us, 3), "dense_gbs": round(dense_bytes / (us * 1e-6) / 1e9, 1),
                               "sparse_us": round(sparse_us, 3), "speedup": round(us / sparse_us, 3)}
                dense_sum[M] += us
                sparse_sum[M] += sparse_us
                del g, y
            out["shapes"][name] = rec
            del ws, w0
            torch.cuda.empty_cache()
        out["launch_sum_speedup"] = {str(M): round(dense_sum[M] / sparse_sum[M], 3) for M in Ms}
        # the dense decode step: the same launch sequence as the sparse step
        layers = [{name: torch.from_numpy(host[name][0].view(np.int16)).to(dev).view(torch.bfloat16)
                   for name in SHAPES}]
        layers += [{name: w.clone() for name, w in layers[0].items()} for _ in range(LAYERS - 1)]
        dense_step = {}
        for M in Ms:
            ys = {name: torch.empty((M, layers[0][name].shape[0]), dtype=torch.bfloat16, device=dev)
                  for name in SHAPES}
            for name in SHAPES:
                torch.matmul(xs[name][:M], layers[0][name].t(), out=ys[name])
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                for lw in layers:
                    for name in SHAPES:
                        torch.matmul(xs[name][:M], lw[name].t(), out=ys[name])
            for _ in range(3):
                g.replay()
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(10):
                g.replay()
            b.record()
            torch.cuda.synchronize()
            dense_step[M] = a.elapsed_time(b) / 10
            del g, ys
        del layers
        torch.cuda.empty_cache()
        out["dense_step_ms"] = {str(M): round(v, 4) for M, v in dense_step.items()}
        out["step_speedup"] = {str(M): round(dense_step[M] / results[M]["step_ms"], 3) for M in Ms}
        buf = torch.zeros(2 ** 28, dtype=torch.float32, device=dev)
        acc = torch.empty((), dtype=torch.float32, device=dev)
        torch.sum(buf, dim=0, out=acc)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(5):
                torch.sum(buf, dim=0, out=acc)
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(10):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        out["read_stream_gbs"] = round(50 * buf.numel() * 4 / (a.elapsed_time(b) * 1e-3) / 1e9, 1)
        out["read_stream_how"] = "torch.sum over a 1 GiB fp32 buffer, CUDA graph of 5, 10 replays"
        del g, buf, acc
        torch.cuda.empty_cache()
    except Exception as e:  # context only: never let it end the run
        out["error"] = repr(e)[:300]
    return out


# The source files that compile into each profiled kernel (its translation unit and the
# device headers it includes, plus the public headers without their comments and function
# prototypes); host-only files such as sp_api.cu do not change the kernel.
KERNEL_SOURCES = {
    "linear_ccw_kernel": ("sp_linear_cc.cu", "sp_cc_common.cuh", "sp_internal.cuh"),
    "linear_cc_kernel": ("sp_linear_cc.cu", "sp_cc_common.cuh", "sp_internal.cuh"),
    "linear_tc_kernel": ("sp_linear_tc.cu", "sp_internal.cuh"),
    "chain_kernel": ("sp_chain.cu", "sp_cc_common.cuh", "sp_internal.cuh"),
}


def kernel_source_hash(kernel: str):
    """Hash of the sources of `kernel`; None for a kernel without a source list."""
    files = KERNEL_SOURCES.get(kernel)
    if files is None:
        return None
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2405_03594_gb300", "csrc")
    for n in files:
        with open(os.path.join(csrc, n)) as f:
            # code only: a comment edit leaves the compiled kernel (and its counters) unchanged
            code = re.sub(r"/\*.*?\*/|//[^\n]*", "", f.read(), flags=re.S)
        h.update(n.encode() + b"\0" + " ".join(code.split()).encode())
    for n in ("sp.h", "sp_stack.h"):
        with open(os.path.join(ROOT, "include", n)) as f:
            code = re.sub(r"/\*.*?\*/|//[^\n]*", "", f.read(), flags=re.S)
        # function prototypes declare host entry points and compile into no kernel
        code = re.sub(r"(?:sp_status|const\s+char\s*\*)\s*sp_\w+\s*\([^;{}]*\)\s*;", "", code)
        h.update(n.encode() + b"\0" + " ".join(code.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the
    current kernel sources; else None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(f"{kernel}|{workload}")
    if not e or e.get("source_hash") is None or e.get("source_hash") != kernel_source_hash(kernel):
        return None
    return e.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.gpu = gpu_index
        self.p = None

    def __enter__(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.p:
            time.sleep(0.2)
            self.p.terminate()
            self.p.wait()

    def summary(self):
        self.f.flush()
        self.f.seek(0)
        rows = [r.strip().split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [c.strip() for c in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx = float(r[2])
            except ValueError:
                continue
            for nm, v in zip(names, r[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


def cpu_oracle_leg(host, M: int, reps_target_s: float = 10.0):
    """Time the float64 oracle on this host's cores on layer 0 (all four linears),
    repeated for about `reps_target_s` seconds (at least three runs), and scale the median
    run to a 32-layer step.  Returns (cpu_baseline dict, oracle outputs)."""
    cores = len(os.sched_getaffinity(0))
    os.environ.setdefault("OMP_NUM_THREADS", str(cores))
    import oracle

    outs = {}
    t_layer = []
    deadline = time.perf_counter() + reps_target_s
    while True:
        t0 = time.perf_counter()
        for name in SHAPES:
            W, mask, x = host[name]
            outs[name] = oracle.linear_bf16(x[:M], W, mask)
        t_layer.append(time.perf_counter() - t0)
        if time.perf_counter() > deadline and len(t_layer) >= 3:
            break
    t = sorted(t_layer)[len(t_layer) // 2]
    return ({"value": M / (LAYERS * t), "unit": "tok/s", "cores": cores, "kind": "oracle",
             "sample": f"layer 0 (qkv, o, gate_up, down) at M={M}, float64 C oracle, OpenMP over rows; "
                       f"median of {len(t_layer)} runs of {t:.2f} s, x{LAYERS} layers"},
            outs)


def run_reference(args):
    """The float64 oracle on the host cores, on the same workload as our arm: one step is
    the full decode step, the four layer-0 linears (qkv, o, gate_up, down) computed for
    each of the 32 layers at M rows -- the same 128 products and the same bytes that our
    arm's step streams (its 32 layers are copies of layer 0 too).  Nothing is sampled or
    extrapolated: the timed region is exactly `steps` such steps."""
    rank, _, world = dist_env()
    if rank != 0:
        return
    host = host_layer(args.pct, args.m)
    cores = len(os.sched_getaffinity(0))
    os.environ.setdefault("OMP_NUM_THREADS", str(cores))
    import oracle

    def step():
        for _ in range(LAYERS):
            for name in SHAPES:
                W, mask, x = host[name]
                oracle.linear_bf16(x[: args.m], W, mask)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    t = (time.perf_counter() - t0) / args.steps
    value = args.m / t
    line = {"metric": METRIC, "value": value, "unit": "tok/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded, Llama-2-7B shapes)", "impl": "reference",
            "config": {"workload": workload_name(args.pct, args.m), "M": args.m},
            "cpu_baseline": {"value": value, "unit": "tok/s", "cores": cores, "kind": "oracle",
                             "sample": f"the whole step: {LAYERS} x (qkv, o, gate_up, down) at M={args.m}, "
                                       f"float64 C oracle, OpenMP over output rows; no extrapolation"},
            "e2e": {"value": value, "unit": "tok/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def workload_name(pct: int, M: int) -> str:
    return (f"llama2-7b {LAYERS}-layer linear stack (qkv 4096->12288, o 4096->4096, gate_up 4096->22016, "
            f"down 11008->4096), {pct}% per-row sparsity, bf16 bitmask format, decode M={M}")


def chain_bytes(cs, M: int) -> int:
    """Algorithmic bytes of one chained step: per linear the compressed values, one mask
    bit per weight, the INT8 scales, x read and y written; residual epilogues also read
    the old y and r."""
    tot = 0
    for mat, x, y, epi, r in cs.ops(M):
        b = algorithmic_bytes(mat.info, M, mat.k, y.shape[1])
        if epi == "residual":
            b += 2 * M * mat.n + 2 * mat.n
        tot += b
    return tot


def time_chain(cs, M: int, steps: int, warmup: int, world: int):
    """Time `steps` decode steps of a ChainStack: each step is the input copy plus one
    sp_chain_run launch; CUDA events bracket the whole run and every chain launch."""
    import torch

    from paper_2405_03594_gb300 import sp, synth

    x = synth.activations(M, 4096, synth.rng(0, 0, 0, synth.STREAM_X))
    cs.set_input(torch.from_numpy(x.view(np.int16)).to(cs.dev).view(torch.bfloat16))
    c = cs.chain(M)
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        cs.step(M)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    evs = []
    t0.record(stream)
    for _ in range(steps):
        sp.copy_columns(cs.h[:M], cs.x0[:M], 0)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        c.run()
        b.record(stream)
        evs.append((a, b))
    t1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    sp.check()
    step_ms = t0.elapsed_time(t1) / steps
    chain_us = sum(a.elapsed_time(b) for a, b in evs) / steps * 1e3
    return step_ms, chain_us


def chained_section(args, peak_gbs, host_bf):
    """The decode step of the 32-layer linear stack with its elementwise glue (residual adds,
    gate*up), bf16 70%, run two ways on the same weights: one sp_chain_run launch per step
    (glue fused into the epilogues) and a CUDA graph of separate launches (sp_linear plus
    the glue kernels).  The chained launch's parity, linear by linear against the float64
    oracle on the GPU's own inputs, is checked by the GPU tests, not here."""
    import torch

    from paper_2405_03594_gb300 import sp, synth
    from paper_2405_03594_gb300.stack import ChainStack, LinearStack

    out = {"workload": f"llama2-7b linear stack decode step, {LAYERS} layers x (qkv, o + residual, gate_up -> "
                       f"gate*up, down + residual), {args.pct}% bf16, N(0, 0.003^2) weights",
           "chain": {}, "graph": {}}
    cs = ChainStack(layers=LAYERS, pct=args.pct, int8=False, max_m=4, host=host_bf)
    for M in (1, 4):
        ms, cu = time_chain(cs, M, max(3, min(args.steps, 100)), max(3, args.warmup), 1)
        b = chain_bytes(cs, M)
        out["chain"][str(M)] = {"tok_s": M / (ms * 1e-3), "ms_per_step": ms, "chain_us": cu,
                                "gbs": b / (cu * 1e-6) / 1e9, "frac_of_peak": b / (cu * 1e-6) / 1e9 / peak_gbs,
                                "launches_per_step": cs.launches_per_step(M), "kernel": "chain_kernel",
                                "activations_finite": bool(torch.isfinite(cs.h[:M].float()).all().item())}
    del cs
    torch.cuda.empty_cache()
    st = LinearStack(layers=LAYERS, pct=args.pct, int8=False, max_m=4, host=host_bf)
    for M in (1, 4):
        x = synth.activations(M, 4096, synth.rng(0, 0, 0, synth.STREAM_X))
        st.set_input(torch.from_numpy(x.view(np.int16)).to(st.dev).view(torch.bfloat16))
        g = st.capture(M)
        ms = time_graph(g, max(3, min(args.steps, 100)), max(3, args.warmup))
        sp.check()
        out["graph"][str(M)] = {"tok_s": M / (ms * 1e-3), "ms_per_step": ms,
                                "launches_per_step": st.launches_per_step(M)}
        del g
    del st
    torch.cuda.empty_cache()
    return out


def run_ours(args):
    import numpy as np
    import torch

    rank, local_rank, world = dist_env()
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    from paper_2405_03594_gb300 import sp, synth

    Ms = sorted({args.m} | {int(v) for v in args.sweep.split(",") if v.strip()})
    Mmax = max(Ms)
    host = host_layer(args.pct, Mmax)
    mats, xs, ys = {}, {}, {}
    for name in SHAPES:
        W, mask, x = host[name]
        h0 = sp.compress(torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16),
                         torch.from_numpy(mask).to(dev))
        mats[name] = [h0] + [h0.clone() for _ in range(LAYERS - 1)]
        xs[name] = torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)
        ys[name] = torch.empty((Mmax, h0.n), dtype=torch.bfloat16, device=dev)
    torch.cuda.synchronize()
    ws_bytes = max(h.workspace_size(Mmax) for h in (mats[n][0] for n in SHAPES))
    ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device=dev)

    def linear(name, layer, M, stream=None):
        mats[name][layer].linear(xs[name][:M], out=ys[name][:M], workspace=ws, path=args.path, stream=stream)

    def per_m(M):
        # per-launch times: one CUDA graph per shape, its 32 layers back to back
        for name in SHAPES:
            linear(name, 0, M)
        torch.cuda.synchronize()
        graphs = {}
        for name in SHAPES:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                for layer in range(LAYERS):
                    linear(name, layer, M)
            graphs[name] = g
        torch.cuda.synchronize()
        stream = torch.cuda.current_stream()
        for _ in range(args.warmup):
            for name in SHAPES:
                graphs[name].replay()
        torch.cuda.synchronize()
        ev = {name: [] for name in SHAPES}
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for _ in range(args.steps):
            for name in SHAPES:
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record(stream)
                graphs[name].replay()
                b.record(stream)
                ev[name].append((a, b))
        t_end.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        shape_ms = {name: sum(a.elapsed_time(b) for a, b in ev[name]) for name in SHAPES}
        sp.check()
        # the decode step itself: the 128 linears in layer order (qkv, o, gate_up, down of
        # layer 0, then layer 1, ...) in one graph; its time is the step time
        gs = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gs):
            for layer in range(LAYERS):
                for name in SHAPES:
                    linear(name, layer, M)
        for _ in range(args.warmup):
            gs.replay()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        t_start.record(stream)
        for _ in range(args.steps):
            gs.replay()
        t_end.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        total_ms = t_start.elapsed_time(t_end)
        sp.check()
        graphs["step"] = gs
        return total_ms, shape_ms, graphs

    results = {}
    peak_gbs, peak_kind = load_peaks()
    for M in Ms:
        if M == args.m:
            with ClockSampler(local_rank) as clk:
                total_ms, shape_ms, graphs = per_m(M)
            clocks = clk.summary()
        else:
            total_ms, shape_ms, graphs = per_m(M)
        del graphs
        step_ms = max_over_ranks([total_ms / args.steps], dev)[0]
        step_bytes = 0
        per_shape = {}
        for name in SHAPES:
            h = mats[name][0]
            b = algorithmic_bytes(h.info, M, h.k, h.n)
            step_bytes += LAYERS * b
            launch_us = shape_ms[name] / (args.steps * LAYERS) * 1e3
            per_shape[name] = {"us_per_launch": launch_us, "algorithmic_bytes": b,
                               "gbs": b / (launch_us * 1e-6) / 1e9, "frac": b / (launch_us * 1e-6) / 1e9 / peak_gbs}
        results[M] = {"step_ms": step_ms, "tok_s": whole_job_tok_s(world, M, step_ms),
                      "step_gbs": step_bytes / (step_ms * 1e-3) / 1e9, "per_shape": per_shape,
                      "step_bytes": step_bytes}

    M = args.m
    r = results[M]
    dom = max(SHAPES, key=lambda n: r["per_shape"][n]["us_per_launch"])
    d = r["per_shape"][dom]
    kern = mats[dom][0].kernel_name(M, args.path)
    workload = f"{dom} {args.pct}% bf16 M={M}"
    roofline = {"bound": "hbm", "achieved": d["gbs"], "peak": peak_gbs, "unit": "GB/s", "frac": d["frac"],
                "traffic": profiled_traffic(kern, workload), "kernel": kern, "launch": workload,
                "peak_kind": f"of {peak_kind}",
                "algorithmic_bytes_per_launch": d["algorithmic_bytes"], "us_per_launch": d["us_per_launch"],
                "frac_of_nominal_8tbs": d["gbs"] / NOMINAL_HBM_GBS}

    # ---------------------------------------------------------------- end to end
    # Public API calls (no graph), inputs copied from pinned host memory every step and
    # the step's result (the last down projection) copied back.
    pinned_x = {name: xs[name][:M].cpu().pin_memory() for name in SHAPES}
    pinned_y = torch.empty((M, mats["down"][0].n), dtype=torch.bfloat16).pin_memory()
    stream = torch.cuda.current_stream()
    e2e_steps = max(3, min(args.steps, 50))

    def e2e_step():
        for name in SHAPES:
            xs[name][:M].copy_(pinned_x[name], non_blocking=True)
        for layer in range(LAYERS):
            for name in SHAPES:
                linear(name, layer, M)
        pinned_y.copy_(ys["down"][:M], non_blocking=True)

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(e2e_steps):
        e2e_step()
    b.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks([a.elapsed_time(b) / e2e_steps], dev)[0]
    h2d = sum(pinned_x[n].numel() * 2 for n in SHAPES)
    d2h = pinned_y.numel() * 2

    # ---------------------------------------------------------------- parity + CPU oracle (rank 0, N=1)
    cpu = None
    parity = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu, outs = cpu_oracle_leg(host, M)
        worst = 0.0
        fro = 0.0
        for name in SHAPES:
            mats[name][0].linear(xs[name][:M], out=ys[name][:M], workspace=ws, path=args.path)
            y = synth.bf16_to_f32(ys[name][:M].view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.float64)
            ref = outs[name]
            worst = max(worst, float(np.abs(y - ref).max() / np.abs(ref).max()))
            fro = max(fro, float(np.linalg.norm(y - ref) / np.linalg.norm(ref)))
        parity = {"max_err_over_max_ref": worst, "rel_fro": fro, "ok": worst <= 1e-2 and fro <= 5e-3}

    # kernel launches per linear of the timed step (the library's own count)
    launch_counts = {name: mats[name][0].launch_count(M, args.path) for name in SHAPES}
    del mats
    torch.cuda.empty_cache()
    sections = {"per_m": {str(m): {"tok_s": v["tok_s"], "step_ms": v["step_ms"], "step_gbs": v["step_gbs"],
                                   "frac_of_peak": v["step_gbs"] / peak_gbs,
                                   "per_shape": {n: {"us": s["us_per_launch"], "gbs": s["gbs"], "frac": s["frac"]}
                                                 for n, s in v["per_shape"].items()}}
                          for m, v in results.items()}}
    host_bf = None
    if world == 1 and not (args.no_chain and args.no_stack):
        from paper_2405_03594_gb300.stack import host_layer as stack_host_layer

        host_bf = stack_host_layer(args.pct, False)
    if world == 1:
        if not args.no_chain:
            sections["chained_step_bf16"] = chained_section(args, peak_gbs, host_bf)
        if not args.no_stack:
            sections["stack_int8"] = stack_section(args, peak_gbs, host_bf)
        if not args.no_prefill:
            sections["prefill"] = prefill_section(args)
        if not args.no_dense:
            sections["dense_comparison"] = dense_section(host, xs, results, Ms)
        if not args.no_update:
            sections["masked_update"] = update_section(args, host, peak_gbs)
        if not args.no_w8a8:
            sections["w8a8"] = w8a8_section(args, host, peak_gbs)
        if not args.no_sweep_config:
            sections["sparsity_batch_sweep"] = sweep_section(args, peak_gbs)
        if not args.no_profile:
            sections["per_layer_profile"] = profile_section(args, peak_gbs)
        if not args.no_square:
            sections["square_12288"] = square_section(args)

    if rank == 0:
        if args.sections_out:
            with open(args.sections_out, "w") as f:
                json.dump(sections, f, indent=1)
        line = headline_line(args, world, r, roofline, {
            "value": whole_job_tok_s(world, M, e2e_ms), "unit": "tok/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h}, cpu, clocks, parity, LAYERS * sum(launch_counts.values()) * args.steps,
            section_summary(sections))
        print(json.dumps(line, separators=(",", ":")), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def _sig(v, n: int = 4):
    """v rounded to n significant digits (None and non-numbers pass through)."""
    if isinstance(v, bool) or not isinstance(v, (int, float)):
        return v
    if v == 0 or v != v:
        return v
    from math import floor, log10

    return round(v, max(0, n - 1 - int(floor(log10(abs(v))))))


def section_summary(sections: dict) -> dict:
    """A few figures of each context section, small enough for the headline line; the
    full sections go to --sections-out."""
    out = {}
    pm = sections.get("per_m") or {}
    if pm:
        out["tok_s_by_m"] = {m: _sig(v["tok_s"]) for m, v in pm.items()}
    ch = sections.get("chained_step_bf16")
    if ch:
        out["chain_bf16_tok_s"] = {m: _sig(v["tok_s"]) for m, v in ch.get("chain", {}).items()}
        out["graph_bf16_tok_s"] = {m: _sig(v["tok_s"]) for m, v in ch.get("graph", {}).items()}
    st = sections.get("stack_int8")
    if st:
        out["stack_int8_tok_s"] = {"graph": {m: _sig(v["tok_s"]) for m, v in st.get("graph_per_m", {}).items()},
                                   "chain": {m: _sig(v["tok_s"]) for m, v in st.get("chain_per_m", {}).items()}}
    pf = sections.get("prefill")
    if pf and pf.get("shapes"):
        fr = {k: v["frac_dense_executed"] for k, v in pf["shapes"].items()}
        out["prefill_frac_dense"] = {"min": _sig(min(fr.values()), 3), "max": _sig(max(fr.values()), 3)}
    up = sections.get("masked_update")
    if up and up.get("shapes"):
        out["update_frac"] = {n: _sig(v["frac"], 3) for n, v in up["shapes"].items()}
    wa = sections.get("w8a8")
    if wa and wa.get("shapes", {}).get("gate_up"):
        # gate_up: time of sp_linear_w8a8 / time of the INT8-weight linear on bf16 x
        out["w8a8_rel"] = {m: _sig(v["w8a8_over_int8_weight"], 3) for m, v in wa["shapes"]["gate_up"].items()
                           if m in ("1", "64")}
    de = sections.get("dense_comparison")
    if de and de.get("step_speedup"):
        out["vs_dense_cublas"] = {m: _sig(v, 3) for m, v in de["step_speedup"].items()}
    sw = sections.get("sparsity_batch_sweep")
    if sw and sw.get("points"):
        out["sweep_frac"] = {k: {m: _sig(p["by_m"][m]["frac_of_roofline"], 2) for m in ("16", "256")
                                 if m in p["by_m"]}
                             for k, p in sw["points"].items() if k.endswith("@70%")}
    pr = sections.get("per_layer_profile")
    if pr and pr.get("chain"):
        out["profile_tok_s"] = {"chain": _sig(pr["chain"]["tok_s"]), "graph": _sig(pr.get("graph", {}).get("tok_s"))}
    sq = sections.get("square_12288")
    if sq and sq.get("points"):
        out["square_speedup_vs_0pct"] = {p: _sig(sq["points"][p]["speedup_vs_0pct"], 3) for p in ("50", "70", "90")
                                         if p in sq["points"]}
    for k in ("chained_step_bf16", "stack_int8", "prefill", "dense_comparison", "masked_update", "w8a8",
              "sparsity_batch_sweep", "per_layer_profile", "square_12288"):
        if sections.get(k) and sections[k].get("error"):
            out.setdefault("errors", {})[k] = str(sections[k]["error"])[:80]
    return out


def headline_line(args, world: int, r: dict, roofline: dict, e2e: dict, cpu, clocks, parity, gpu_launches: int,
                  summary: dict) -> dict:
    """The one JSON line bench.py prints: the contract's keys, the roofline of the dominant
    kernel, the CPU baseline, the clocks seen while timing, and a compact summary of the
    context sections (kept to about 2 KB so that the whole line survives a tail capture)."""
    M = args.m
    rf = {k: _sig(v) for k, v in roofline.items()}
    line = {
        "metric": METRIC, "value": _sig(r["tok_s"], 6), "unit": "tok/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": _sig(r["step_ms"], 6), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: seeded N(0,0.02^2) W, per-row magnitude masks, N(0,1) x; 32 copies of layer 0",
        "config": {"workload": workload_name(args.pct, M), "M": M, "layers": LAYERS, "sparsity_pct": args.pct,
                   "path": args.path,
                   "l2": f"no flush: {r['step_bytes'] / 1e9:.2f} GB of distinct weights per step",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "e2e": {k: _sig(v, 6) for k, v in e2e.items()},
        "gpu_launches": gpu_launches,
        "roofline": rf,
        "cpu_baseline": None if cpu is None else {k: _sig(v) for k, v in cpu.items()},
        "clocks": clocks,
        "step_gbs": _sig(r["step_gbs"]),
        "parity_layer0": None if parity is None else {k: _sig(v, 3) for k, v in parity.items()},
        "summary": summary,
    }
    return line


def run_single(args):
    """One linear of one shape, launched directly, or the chained step of --layers layers:
    a small case for ncu captures."""
    import torch

    if args.single == "chain":
        from paper_2405_03594_gb300.stack import ChainStack

        cs = ChainStack(layers=args.layers, pct=args.pct, int8=False, max_m=4)
        ms, us = time_chain(cs, args.m, max(args.steps, 1), args.warmup, 1)
        nbytes = chain_bytes(cs, args.m)
        print(json.dumps({"single": "chain", "layers": args.layers, "M": args.m, "pct": args.pct,
                          "us_per_launch": us, "step_ms": ms, "algorithmic_bytes": nbytes,
                          "gbs": nbytes / (us * 1e-6) / 1e9}), flush=True)
        return

    from paper_2405_03594_gb300 import sp, synth

    dev = torch.device("cuda", 0)
    W, mask, x = synth.layer_inputs(args.single, args.pct, args.m, seed=0, layer=0)
    if args.int8:
        q, sc = synth.quantize_int8(W, mask)
        h = sp.compress(torch.from_numpy(q).to(dev), torch.from_numpy(mask).to(dev), torch.from_numpy(sc).to(dev))
    else:
        h = sp.compress(torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16),
                        torch.from_numpy(mask).to(dev))
    if args.update:
        run_single_update(args, h, mask, dev)
        return
    xd = torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)
    y = torch.empty((args.m, h.n), dtype=torch.bfloat16, device=dev)
    ws = torch.zeros(max(h.workspace_size(args.m), 256), dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        h.linear(xd, out=y, workspace=ws, path=args.path)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        h.linear(xd, out=y, workspace=ws, path=args.path)
    b.record()
    torch.cuda.synchronize()
    sp.check()
    us = a.elapsed_time(b) / max(args.steps, 1) * 1e3
    nbytes = algorithmic_bytes(h.info, args.m, h.k, h.n)
    print(json.dumps({"single": args.single, "M": args.m, "pct": args.pct, "int8": args.int8, "us_per_launch": us,
                      "algorithmic_bytes": nbytes, "gbs": nbytes / (us * 1e-6) / 1e9}), flush=True)


def square_section(args) -> dict:
    """The 12288 x 12288 sparse matmul against sparsity (the scaling example of Sec. 2.3, there
    on a CS-3; here on the tensor-core kernel): x [2048, 12288] bf16, per-row magnitude masks at
    0, 10, ..., 90 %, y = x . (W o M)^T.  Per sparsity the launch time, its speedup over the 0 %
    matrix through the same kernel, the ideal 1 / (1 - s), and the speedup over the dense cuBLAS
    GEMM of the same shape.  Parity of this shape is checked by the GPU tests.  A failure is
    reported in the section instead of ending the run."""
    import torch

    from paper_2405_03594_gb300 import sp, synth

    out = {"what": "12288 x 12288, M = 2048, tensor-core kernel, per-row magnitude masks", "N": 12288, "K": 12288,
           "M": 2048, "kernel": "linear_tc_kernel", "points": {}}
    try:
        dev = torch.device("cuda", 0)
        N = K = 12288
        M = 2048
        W = synth.weight(N, K, synth.rng(0, 0, 0, synth.STREAM_W))
        x = synth.activations(M, K, synth.rng(0, 0, 0, synth.STREAM_X))
        xd = torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)
        y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
        reps = max(3, min(args.steps, 20))

        def timed(fn):
            for _ in range(3):
                fn()
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(reps):
                fn()
            b.record()
            torch.cuda.synchronize()
            return a.elapsed_time(b) / reps * 1e3

        Wd = torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16)
        dense_us = timed(lambda: torch.matmul(xd, Wd.t()))
        out["dense_cublas_us"] = dense_us
        base = None
        for pct in range(0, 100, 10):
            mask = synth.magnitude_mask(W, pct)
            h = sp.compress(Wd, torch.from_numpy(mask).to(dev))
            ws = torch.zeros(max(h.workspace_size(M), 256), dtype=torch.uint8, device=dev)
            us = timed(lambda: h.linear(xd, out=y, workspace=ws, path="tensor_core"))
            sp.check()
            base = us if base is None else base
            out["points"][str(pct)] = {"us": us, "speedup_vs_0pct": base / us, "ideal": 1.0 / (1.0 - pct / 100.0),
                                       "speedup_vs_dense_cublas": dense_us / us, "nnz": int(h.info.nnz),
                                       "compressed_bytes": int(h.info.bytes)}
            del h, ws
            torch.cuda.empty_cache()
    except Exception as e:  # context only: never let it end the run
        out["error"] = f"{type(e).__name__}: {e}"
    return out


def run_square_sweep(args):
    """Only the 12288 x 12288 sweep (--square-sweep): one JSON line."""
    print(json.dumps({"single": "square_sweep", **square_section(args)}), flush=True)


def profile_section(args, peak_gbs) -> dict:
    """The 32-layer bf16 decode step with a per-layer sparsity profile (60 .. 80 %, mean 70 %;
    the stand-in for an outlier-weighted layerwise profile): one chained launch per step and a
    CUDA graph of separate launches, at M = 1, beside the uniform 70 % step of the chained
    section.  Every layer's masks are drawn at its own sparsity from the seeded layer-0 weights
    (the five levels' masks, one per shape and level).  Parity of such profiles, linear by
    linear through both paths, is checked by the GPU tests.  A failure is reported in the
    section instead of ending the run."""
    import torch

    from paper_2405_03594_gb300 import sp, synth
    from paper_2405_03594_gb300.stack import STACK_WEIGHT_STD, ChainStack, LinearStack

    prof = synth.layer_sparsity_profile(LAYERS)
    out = {"profile": prof, "mean_pct": sum(prof) / len(prof), "M": 1}
    try:
        if not torch.cuda.is_available():
            raise RuntimeError("no CUDA device")
        levels = sorted(set(prof))
        per_level = {p: synth.stack_layer(p, False, seed=0, layer=0, std=STACK_WEIGHT_STD) for p in levels}
        hosts = [per_level[p] for p in prof]
        cs = ChainStack(int8=False, max_m=1, host_layers=hosts)
        ms, cu = time_chain(cs, 1, max(3, min(args.steps, 100)), max(3, args.warmup), 1)
        b = chain_bytes(cs, 1)
        out["chain"] = {"tok_s": 1 / (ms * 1e-3), "ms_per_step": ms, "chain_us": cu, "gbs": b / (cu * 1e-6) / 1e9,
                        "frac_of_peak": b / (cu * 1e-6) / 1e9 / peak_gbs, "weight_bytes": cs.weight_bytes()}
        del cs
        torch.cuda.empty_cache()
        st = LinearStack(int8=False, max_m=1, host_layers=hosts)
        x = synth.activations(1, 4096, synth.rng(0, 0, 0, synth.STREAM_X))
        st.set_input(torch.from_numpy(x.view(np.int16)).to(st.dev).view(torch.bfloat16))
        g = st.capture(1)
        ms = time_graph(g, max(3, min(args.steps, 100)), max(3, args.warmup))
        sp.check()
        out["graph"] = {"tok_s": 1 / (ms * 1e-3), "ms_per_step": ms, "launches_per_step": st.launches_per_step(1)}
        del g, st
        torch.cuda.empty_cache()
    except Exception as e:  # context only: never let it end the run
        out["error"] = f"{type(e).__name__}: {e}"
    return out


def update_bytes(mask: np.ndarray, info) -> int:
    """Algorithmic bytes of one masked update: the 32-byte gradient sectors (8 float32
    columns) that hold at least one kept column, the kept values read and written, the
    masks, and the chunk offsets."""
    N, K = mask.shape
    sectors = int(np.count_nonzero(mask.reshape(N, K // 8, 8).any(axis=2)))
    return 32 * sectors + 2 * 2 * int(info.nnz) + N * K // 8 + 8 * (int(info.tiles * info.row_blocks) + 1)


SWEEP_SHAPES = ("gate_up", "down")
SWEEP_PCTS = (0, 50, 60, 70, 80)
SWEEP_MS = (1, 2, 4, 8, 16, 32, 64, 128, 256)


def sweep_copies(compressed_bytes: int) -> int:
    """Distinct device copies of one matrix so that a graph of launches over them reads
    more than 3x L2 of compressed weights (no L2 flush needed between launches)."""
    return max(2, -(-int(3 * L2_BYTES) // max(int(compressed_bytes), 1)))


def roofline_time_us(nbytes: int, nnz: int, M: int, hbm_gbs: float, tensor_tflops: float) -> tuple[float, str]:
    """The slower of the compressed bytes over the HBM peak and the nonzero FLOPs
    (2 M nnz) over the bf16 tensor peak, in microseconds, and which one it is."""
    t_bytes = nbytes / (hbm_gbs * 1e9) * 1e6
    t_flops = 2.0 * M * nnz / (tensor_tflops * 1e12) * 1e6
    return (t_bytes, "hbm") if t_bytes >= t_flops else (t_flops, "tensor")


def sweep_section(args, peak_gbs):
    """The sparsity x batch sweep: gate_up 4096->22016 and down 11008->4096, non-uniform
    masks (per-row sparsity within +-10 points of the target, 5% dense input columns) at
    0/50/60/70/80%, M = 1 ... 256 on the automatic kernel choice.  Each point is a CUDA graph
    of launches over enough distinct copies to read > 3x L2; per-launch time, GB/s, and the
    fraction of the roofline (the slower of bytes over HBM peak and nonzero FLOPs over the
    bf16 tensor peak).  Parity of the same inputs is checked by the GPU tests."""
    import torch

    from paper_2405_03594_gb300 import sp, synth

    tensor_peak, tkind = load_tensor_peak()
    dev = torch.device("cuda", 0)
    res = {"workload": "gate_up 4096->22016 and down 11008->4096, non-uniform per-row magnitude masks "
                       "(+-10 points, 5% dense columns), bf16, auto kernel",
           "hbm_peak_gbs": peak_gbs, "tensor_peak_tflops": tensor_peak, "tensor_peak_kind": tkind, "points": {}}
    try:
        for name in SWEEP_SHAPES:
            N, K = synth.LLAMA2_7B_SHAPES[name]
            p = synth.PROJ_IDS[name]
            W = synth.weight(N, K, synth.rng(0, 0, p, synth.STREAM_W))
            x = synth.activations(max(SWEEP_MS), K, synth.rng(0, 0, p, synth.STREAM_X))
            xd = torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)
            Wd = torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16)
            for pct in SWEEP_PCTS:
                mask, _, _ = synth.nonuniform_mask(W, pct, synth.rng(0, 0, p, synth.STREAM_MASK))
                h0 = sp.compress(Wd, torch.from_numpy(mask).to(dev))
                copies = sweep_copies(int(h0.info.bytes))
                hs = [h0] + [h0.clone() for _ in range(copies - 1)]
                y = torch.empty((max(SWEEP_MS), N), dtype=torch.bfloat16, device=dev)
                ws = torch.zeros(max(max(h0.workspace_size(M) for M in SWEEP_MS), 256), dtype=torch.uint8, device=dev)
                pts = {}
                for M in SWEEP_MS:
                    for h in hs:
                        h.linear(xd[:M], out=y[:M], workspace=ws)
                    torch.cuda.synchronize()
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(g):
                        for h in hs:
                            h.linear(xd[:M], out=y[:M], workspace=ws)
                    ms = time_graph(g, 10, 3)
                    sp.check()
                    us = ms * 1e3 / copies
                    nbytes = algorithmic_bytes(h0.info, M, K, N)
                    t_roof, bound = roofline_time_us(nbytes, int(h0.info.nnz), M, peak_gbs, tensor_peak)
                    pts[str(M)] = {"us": us, "tok_s": M / (us * 1e-6), "gbs": nbytes / (us * 1e-6) / 1e9,
                                   "tflops_nonzero": 2.0 * M * int(h0.info.nnz) / (us * 1e-6) / 1e12,
                                   "bound": bound, "frac_of_roofline": t_roof / us,
                                   "kernel": h0.kernel_name(M)}
                    del g
                res["points"][f"{name}@{pct}%"] = {"copies": copies, "nnz": int(h0.info.nnz),
                                                   "compressed_bytes": int(h0.info.bytes), "by_m": pts}
                del hs, h0, y, ws
                torch.cuda.empty_cache()
            del Wd, xd
    except Exception as e:  # context only: never let it end the run
        res["error"] = f"{type(e).__name__}: {e}"
    torch.cuda.empty_cache()
    return res


def w8a8_section(args, host, peak_gbs):
    """INT8 weights with INT8 activations (sp_linear_w8a8: per-token absmax x, widened to bf16
    by one launch, then the INT8-weight linear) against the INT8-weight linear alone on bf16
    x, gate_up and down at the bench's sparsity, M = 1 / 16 / 64; back-to-back calls over
    enough distinct copies of the compressed matrix to exceed 3x L2.  Context next to the
    decode step; a failure is reported in the section and never ends the run."""
    import torch

    from paper_2405_03594_gb300 import sp, synth

    dev = torch.device("cuda", 0)
    res = {"what": "sp_linear_w8a8 (2 launches) vs sp_linear on INT8 weights with bf16 x", "shapes": {}}
    try:
        for name in ("gate_up", "down"):
            W, mask, _ = host[name]
            q, sc = synth.quantize_int8(W, mask)
            h0 = sp.compress(torch.from_numpy(q).to(dev), torch.from_numpy(mask).to(dev),
                             torch.from_numpy(sc).to(dev))
            copies = max(2, int(-(-3 * L2_BYTES // int(h0.info.bytes))))
            hs = [h0] + [h0.clone() for _ in range(copies - 1)]
            rec = {}
            for M in (1, 16, 64):
                x = synth.activations(M, h0.k, synth.rng(0, 0, 7, synth.STREAM_X))
                qx, sx = synth.quantize_activations_int8(x)
                qxd, sxd = torch.from_numpy(qx).to(dev), torch.from_numpy(sx).to(dev)
                xd = torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)
                y = torch.empty((M, h0.n), dtype=torch.bfloat16, device=dev)
                ws = torch.zeros(max(h0.w8a8_workspace_size(M), h0.workspace_size(M), 256), dtype=torch.uint8,
                                 device=dev)

                def timed(fn):
                    for h in hs:
                        fn(h)
                    torch.cuda.synchronize()
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    reps = 10
                    a.record()
                    for _ in range(reps):
                        for h in hs:
                            fn(h)
                    b.record()
                    torch.cuda.synchronize()
                    sp.check()
                    return a.elapsed_time(b) / (reps * len(hs)) * 1e3

                us_w8a8 = timed(lambda h: h.linear_w8a8(qxd, sxd, out=y, workspace=ws))
                us_w8 = timed(lambda h: h.linear(xd, out=y, workspace=ws))
                nbytes = (int(h0.info.nnz) + h0.n * h0.k // 8 + int(h0.info.scale_bytes) + M * h0.k + 4 * M
                          + 2 * M * h0.n)
                rec[str(M)] = {"w8a8_us": round(us_w8a8, 3), "int8_weight_us": round(us_w8, 3),
                               "w8a8_over_int8_weight": round(us_w8a8 / us_w8, 3),
                               "w8a8_gbs": round(nbytes / (us_w8a8 * 1e-6) / 1e9, 1),
                               "w8a8_frac": round(nbytes / (us_w8a8 * 1e-6) / 1e9 / peak_gbs, 3),
                               "launches": 2}
                del y, ws
            res["shapes"][name] = rec
            del hs, h0
            torch.cuda.empty_cache()
    except Exception as e:  # context only: never let it end the run
        res["error"] = f"{type(e).__name__}: {e}"[:300]
    return res


def update_section(args, host, peak_gbs):
    """Masked weight update (Algorithm 1's step on the compressed form) on the layer-0
    weights of the four shapes: back-to-back sp_masked_update launches; the float32
    gradients (4 bytes per weight) are larger than L2.  Context next to the decode step;
    a failure here is reported in the section and never ends the run."""
    import torch

    from paper_2405_03594_gb300 import sp

    dev = torch.device("cuda", 0)
    res = {"kernel": "masked_update_kernel", "lr": 1e-3, "peak_gbs": peak_gbs, "shapes": {}}
    try:
        for name in SHAPES:
            W, mask, _ = host[name]
            h = sp.compress(torch.from_numpy(W.view(np.int16)).to(dev).view(torch.bfloat16),
                            torch.from_numpy(mask).to(dev))
            g = torch.randn((h.n, h.k), dtype=torch.float32, device=dev,
                            generator=torch.Generator(dev).manual_seed(0))
            for _ in range(3):
                h.masked_update(g, 1e-3)
            torch.cuda.synchronize()
            reps = 20
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(reps):
                h.masked_update(g, 1e-3)
            b.record()
            torch.cuda.synchronize()
            sp.check()
            us = a.elapsed_time(b) / reps * 1e3
            nbytes = update_bytes(mask, h.info)
            gbs = nbytes / (us * 1e-6) / 1e9
            res["shapes"][name] = {"us": us, "algorithmic_bytes": nbytes, "gbs": gbs, "frac": gbs / peak_gbs}
            del h, g
        torch.cuda.empty_cache()
    except Exception as e:  # context only: never let it end the run
        res["error"] = f"{type(e).__name__}: {e}"
    return res


def run_single_update(args, h, mask, dev):
    """sp_masked_update on one shape, back to back; the float32 gradient (4 bytes per
    weight) is larger than L2 for every Llama-2-7B shape, so no flush is needed."""
    import torch

    from paper_2405_03594_gb300 import sp

    if h.dtype != "bf16":
        raise SystemExit("--update takes bf16 weights only")
    g = torch.randn((h.n, h.k), dtype=torch.float32, device=dev, generator=torch.Generator(dev).manual_seed(0))
    lr = 1e-3
    for _ in range(args.warmup):
        h.masked_update(g, lr)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        h.masked_update(g, lr)
    b.record()
    torch.cuda.synchronize()
    sp.check()
    us = a.elapsed_time(b) / max(args.steps, 1) * 1e3
    nbytes = update_bytes(mask, h.info)
    peak, kind = load_peaks()
    gbs = nbytes / (us * 1e-6) / 1e9
    print(json.dumps({"single": args.single, "op": "masked_update", "pct": args.pct, "us_per_launch": us,
                      "algorithmic_bytes": nbytes, "gbs": gbs, "frac": gbs / peak, "peak_gbs": peak,
                      "peak_kind": kind}), flush=True)


def main():
    args = parse()
    if args.square_sweep:
        run_square_sweep(args)
        return
    if args.single:
        run_single(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
