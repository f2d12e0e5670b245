#!/usr/bin/env python
"""Benchmark: effective TFLOP/s and % of roofline for block-sparse DeiT linears on GB300.

Workload (one "step" = one pass of the whole block-sparse path over one batch): the 12-layer
DeiT-B linear stack (48 GEMMs: qkv 768->2304, proj 768->768, fc1 768->3072 + GELU,
fc2 3072->768) at batch 256 (M = 50432 tokens), 32x32 blocks, per-GEMM block sparsity drawn
U[30%, 70%] as antithetic layer pairs (mean exactly 50%); every weight is packed (mask -> BSR +
work list) and every linear runs, chained layer to layer: by default as one lpvit_bsr_linear_chain
call (the 48 linears in one persistent launch), or with --launch per-linear one call per linear.
Inputs are seeded synthetic bf16 tensors resident in HBM; each step streams ~15 GB, far more than
the 129 MB L2, so no flush is needed.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl lpvit|reference] [--launch chain|per-linear]

Prints one JSON line (rank 0). ``--impl reference`` times the CPU oracle (fp64 C loops on the
host cores) on a bounded row sample of the same workload.
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

METRIC = "effective TFLOP/s and % of roofline for block-sparse DeiT linears"
UNIT = "TFLOP/s"
M_TOKENS = 50432          # DeiT-B, batch 256 x 197 tokens
BLOCK = 32
CONFIG_ID = 4             # seeds of the 12-layer stack workload
WORKLOAD = "deit_b_12layer_linear_stack_batch256"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# GB300 datasheet figures, reported beside the measured denominators: dense bf16 tensor throughput
# (without 2:4 sparsity) and HBM3e bandwidth
NOMINAL_BF16_TFLOPS = 2250.0
NOMINAL_HBM_GBS = 8000.0
PROFILE_TRAFFIC = os.path.join(ROOT, "profiles", "bsr_linear_deit_b_stack_traffic.txt")
# single GEMMs of the stack's shapes (profiling cases): (k, n, b, sparsity, gelu, m)
CASES = {
    "fc1": (768, 3072, 32, 0.5, True, M_TOKENS),
    "fc2": (3072, 768, 32, 0.5, False, M_TOKENS),
    "qkv": (768, 2304, 32, 0.5, False, M_TOKENS),
    "proj": (768, 768, 32, 0.5, False, M_TOKENS),
}

# named workload configurations, one line per GEMM (--config); the seeds follow the parity tests
CONFIG_NAMES = {
    1: "deit_s_qkv_batch1_b32_s50",
    2: "deit_s_layer_batch64_b16_s50",
    3: "deit_b_mlp_batch256_b32_sparsity_sweep",
    5: "deit_b_mlp_zipf1.2_s60_b16_b64_batch1024_and_batch1",
    7: "table2_nonsquare_deit_b_64x32_batch256_and_deit_s_16x32_batch64",
}


def config_gemms(config: int):
    """(label, config, gemm index, m, k, n, block, sparsity, gelu, mask kind) of every GEMM of a
    named configuration; gemm indices as in tests/test_gpu_configs.py."""
    from paper_2407_02068_gb300 import inputs
    out = []
    if config == 1:
        out.append(("qkv", 1, 0, 197, 384, 1152, 32, 0.5, False, "uniform"))
    elif config == 2:
        for g, (name, k, n, gelu) in enumerate(inputs.deit_gemms(inputs.DEIT_S)):
            out.append((name, 2, g, 64 * 197, k, n, 16, 0.5, gelu, "uniform"))
    elif config == 3:
        for s_idx, sp in enumerate([0.0, 0.3, 0.5, 0.7, 0.8]):
            for t in (0, 1):
                k, n, gelu = (768, 3072, True) if t == 0 else (3072, 768, False)
                out.append((f"{'fc1' if t == 0 else 'fc2'}@{sp:.1f}", 3, 2 * s_idx + t, 50432, k, n, 32, sp, gelu,
                            "uniform"))
    elif config == 5:
        for m in (201728, 197):
            for b in (16, 64):
                for t in (0, 1):
                    k, n, gelu = (768, 3072, True) if t == 0 else (3072, 768, False)
                    out.append((f"{'fc1' if t == 0 else 'fc2'}_b{b}_m{m}", 5, t + 2 * (b == 64) + 4 * (m == 197), m,
                                k, n, b, 0.6, gelu, "zipf"))
    elif config == 7:
        for g, (name, k, n, gelu) in enumerate(inputs.deit_gemms(inputs.DEIT_B)):
            out.append((f"deit_b_{name}_64x32", 7, g, 256 * 197, k, n, (64, 32), 0.615, gelu, "uniform"))
        for g, (name, k, n, gelu) in enumerate(inputs.deit_gemms(inputs.DEIT_S)):
            out.append((f"deit_s_{name}_16x32", 7, 4 + g, 64 * 197, k, n, (16, 32), 0.287, gelu, "uniform"))
    return out


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=400)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["lpvit", "reference"], default="lpvit")
    p.add_argument("--e2e-steps", type=int, default=None)
    p.add_argument("--cpu-budget-s", type=float, default=15.0, help="CPU seconds for the oracle baseline sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-dense", action="store_true")
    p.add_argument("--launch", choices=["chain", "per-linear"], default="chain",
                   help="the stack's 48 linears as one lpvit_bsr_linear_chain call (one persistent launch), "
                        "or one lpvit_bsr_linear[_gelu] call each")
    p.add_argument("--case", default="stack", choices=["stack"] + sorted(CASES),
                   help="stack (the benchmarked workload) or one GEMM of it, for profiling")
    p.add_argument("--calibrate", action="store_true",
                   help="fit measured GEMM time to the block-tile count of the paper's power model")
    p.add_argument("--alloc", action="store_true",
                   help="pruning-ratio allocation: distortion curves of the 48 DeiT-B weights + lambda search")
    p.add_argument("--alloc-samples", type=int, default=16, help="per-sample gradients per layer (--alloc)")
    p.add_argument("--alloc-streams", type=int, default=8,
                   help="CUDA streams the 48 independent weights are spread over (--alloc)")
    p.add_argument("--encoder", choices=["deit_b", "deit_s"], default=None,
                   help="end-to-end encoder forward (LayerNorm, attention, block-sparse linears) against dense")
    p.add_argument("--images", type=int, default=256, help="batch of 197-token images (--encoder)")
    p.add_argument("--config", type=int, choices=sorted(CONFIG_NAMES), default=None,
                   help="one JSON line per GEMM of a named workload configuration (L2 flushed and warm, "
                        "CUDA graph at batch 1, binding roofline)")
    p.add_argument("--min-ms", type=float, default=300.0, help="timed wall time per GEMM and mode (--config)")
    return p.parse_args()


# ----------------------------------------------------------------------------------------- helpers

def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    for name in ("lpvit_linear.cu", "lpvit_device.cuh"):
        with open(os.path.join(ROOT, "paper_2407_02068_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(key: str = "dram_bytes_per_stack_linear_launch"):
    """DRAM bytes per launch of the linear kernel (per chain launch: key dram_bytes_per_chain_launch)
    from the committed ncu summary, if it was taken on the current kernel source (else None)."""
    try:
        kv = {}
        with open(PROFILE_TRAFFIC) as f:
            for line in f:
                if ":" in line and not line.startswith("#"):
                    k, v = line.split(":", 1)
                    kv[k.strip()] = v.strip()
        if kv.get("kernel_source_sha") != kernel_source_hash():
            return None
        return float(kv[key])
    except (OSError, KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi clock / throttle sampling every 200 ms while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, smax, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                pw.append(float(parts[3]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "power_w_median": statistics.median(pw) if pw else None, "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def rank_input_seed(rank: int) -> int:
    """Seed of the activations of rank ``rank``: every rank runs its own batch (weak scaling)."""
    from paper_2407_02068_gb300 import inputs
    return inputs.seed(CONFIG_ID, 0, "X") + 7 * rank


def weak_scaling_value(flops_per_rank_step: float, steps: int, world: int, elapsed_max_ms: float) -> float:
    """Whole-job TFLOP/s: the effective FLOPs all ranks processed over the slowest rank's time."""
    return flops_per_rank_step * steps * world / (elapsed_max_ms / 1e3) / 1e12


# ------------------------------------------------------------------------------------ CPU oracle

def oracle_layers_from(stack_layers):
    """Host copies (bf16 bits, masks, biases) of the stack for the oracle."""
    from paper_2407_02068_gb300 import inputs
    out = []
    for L in stack_layers:
        out.append({name: (inputs.bf16_bits(L[name]["W"]), L[name]["mask"].cpu().numpy().astype("uint8"),
                           L[name]["bias"].cpu().numpy(), L[name]["b"]) for name in ("qkv", "proj", "fc1", "fc2")})
    return out


def oracle_step(olayers, h_rows, nthreads):
    """One oracle pass over a row sample: pack every weight, then the chained stack on the rows."""
    import oracle
    for L in olayers:
        for name in ("qkv", "proj", "fc1", "fc2"):
            W, Mk, _, b = L[name]
            oracle.pack(W, Mk, b)
    return oracle.deit_stack_rows(h_rows, olayers, nthreads)


def eff_flops_rows(olayers, rows):
    return sum(2 * rows * int((L[n][1] != 0).sum()) * L[n][3] ** 2 for L in olayers for n in L)


def calibrate_rows(olayers, h_bits, nthreads, budget_s, steps):
    """Rows per oracle step so that `steps` steps (pack + chain) take about `budget_s` seconds."""
    import oracle
    t0 = time.perf_counter()
    for L in olayers:
        for name in ("qkv", "proj", "fc1", "fc2"):
            W, Mk, _, b = L[name]
            oracle.pack(W, Mk, b)
    t_pack = time.perf_counter() - t0
    r0 = min(len(h_bits), max(1, nthreads))
    t0 = time.perf_counter()
    oracle.deit_stack_rows(h_bits[:r0], olayers, nthreads)
    rate = r0 / max(time.perf_counter() - t0, 1e-6)          # rows per second on all threads
    per_step = budget_s / max(steps, 1) - t_pack
    rows = int(max(per_step, 0.0) * rate)
    if rows >= nthreads:
        rows -= rows % nthreads
    return max(1, min(len(h_bits), rows))


def run_reference(args, world, rank):
    """The reference arm: the CPU oracle as it stands, on this host's cores, bounded sample per step."""
    if rank != 0:
        return
    import numpy as np
    import oracle
    from paper_2407_02068_gb300 import inputs
    oracle.build()
    layers = inputs.deit_b_stack(CONFIG_ID, BLOCK, "cpu")
    olayers = oracle_layers_from(layers)
    cores = os.cpu_count() or 1
    total = args.warmup + args.steps
    budget = min(150.0, 6.0 * total)  # whole run within a few minutes
    h_all = inputs.bf16_bits(inputs.activations(4096, 768, inputs.seed(CONFIG_ID, 0, "X")))
    rows = calibrate_rows(olayers, h_all, cores, budget, total)
    rng = np.random.default_rng(0)
    for _ in range(args.warmup):
        oracle_step(olayers, h_all[rng.choice(len(h_all), rows, replace=False)], cores)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(olayers, h_all[rng.choice(len(h_all), rows, replace=False)], cores)
    dt = time.perf_counter() - t0
    flops = eff_flops_rows(olayers, rows) * args.steps
    value = flops / dt / 1e12
    sample = (f"{rows} token rows per step through all 48 GEMMs (+ packing all 48 weights) of the batch-256 "
              f"DeiT-B stack, fp64 C oracle, {cores} threads")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, "M": M_TOKENS, "block": BLOCK, "gemms": 48,
                                            "sample_rows_per_step": rows},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------ GPU arm

def run_gpu(args, world, rank, local):
    import torch
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2407_02068_gb300 import inputs
    from paper_2407_02068_gb300.stack import DeitLinearStack

    layers = inputs.deit_b_stack(CONFIG_ID, BLOCK, dev)
    stack = DeitLinearStack(M_TOKENS, layers, dev)
    # each rank works on its own batch (weak scaling: per-GPU work fixed); weights are replicated
    h0 = inputs.activations(M_TOKENS, 768, rank_input_seed(rank), dev)
    stack.h_in.copy_(h0)
    s = torch.cuda.current_stream()
    ngemm = len(stack.gemms)
    chain = args.launch == "chain"
    nev = 1 if chain else ngemm  # event pairs per step: one per library call

    for _ in range(max(args.warmup, 3)):
        stack.step(chain=chain)
    stack.check()
    torch.cuda.synchronize()

    # ---------------- timed region: K steps, bracketed by two events on the launching stream
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    start.record(s)
    for k in range(args.steps):
        stack.step(chain=chain)
    end.record(s)
    torch.cuda.synchronize()
    # ---------------- the linear kernel's launch durations (roofline): K more steps with an event
    # pair around every library call, i.e. every linear or the chain call (the records cost the
    # stream time, so they stay out of the step time)
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nev)]
          for _ in range(args.steps)]
    ev_step = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
    for k in range(args.steps):
        ev_step[k][0].record(s)
        stack.step(events=ev[k], chain=chain)
        ev_step[k][1].record(s)
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop()
    stack.check()
    elapsed_ms = start.elapsed_time(end)
    lin_ms = sum(a.elapsed_time(b) for row in ev for (a, b) in row)
    # the same pass split three ways: pack (step start to the first linear), the linears, and the
    # gaps between consecutive linears (the rest of that pass's step)
    pack_ms = sum(a.elapsed_time(row[0][0]) for (a, _), row in zip(ev_step, ev))
    evpass_ms = sum(a.elapsed_time(b) for (a, b) in ev_step)
    elapsed_max = max_over_ranks(elapsed_ms, world, dev)
    flops_step = stack.effective_flops()
    value = weak_scaling_value(flops_step, args.steps, world, elapsed_max)
    lin_flops = flops_step * args.steps
    achieved = lin_flops / (lin_ms / 1e3) / 1e12
    peaks, peak_src = load_peaks()
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    peak_sustained = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    traffic = profiled_traffic("dram_bytes_per_chain_launch" if chain else "dram_bytes_per_stack_linear_launch")
    linear_launches = ((ngemm + 47) // 48 if chain else ngemm) * args.steps

    # ---------------- e2e through the public API: pinned host in, pinned host out, every step
    # Each step copies its input from pinned host memory and its result back to pinned host memory,
    # on a copy stream that overlaps the compute stream: step k+1's input goes in once step k's first
    # linear (the only reader of h_in) is done; the result is staged by a device copy on the compute
    # stream (counted in the step) and copied out while the next step runs. The timed region ends
    # when the last result is in host memory.
    e2e_steps = args.e2e_steps or max(10, min(args.steps, 100))
    h0_host = h0.cpu().pin_memory()
    out_host = torch.empty_like(h0_host).pin_memory()
    stage = torch.empty_like(stack.out)
    cs = torch.cuda.Stream(device=dev)
    lin_ev = [(torch.cuda.Event(), torch.cuda.Event()) for _ in range(nev)]
    in_ready, out_ready, out_done = torch.cuda.Event(), torch.cuda.Event(), torch.cuda.Event()

    def e2e_run(nsteps):
        # copy stream, in order: in(0), then per step k: in(k+1) once step k's first linear (the only
        # reader of h_in) is done, out(k) once step k's result is staged
        cs.wait_stream(s)
        with torch.cuda.stream(cs):
            stack.h_in.copy_(h0_host, non_blocking=True)
            in_ready.record(cs)
            out_done.record(cs)
        for k in range(nsteps):
            s.wait_event(in_ready)
            out = stack.step(events=lin_ev, chain=chain)
            if k + 1 < nsteps:
                cs.wait_event(lin_ev[0][1])
                with torch.cuda.stream(cs):
                    stack.h_in.copy_(h0_host, non_blocking=True)
                    in_ready.record(cs)
            s.wait_event(out_done)  # the stage's previous result is in host memory
            stage.copy_(out, non_blocking=True)
            out_ready.record(s)
            cs.wait_event(out_ready)
            with torch.cuda.stream(cs):
                out_host.copy_(stage, non_blocking=True)
                out_done.record(cs)
        s.wait_event(out_done)

    e2e_run(2)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    e0.record(s)
    e2e_run(e2e_steps)
    e1.record(s)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    e2e_value = weak_scaling_value(flops_step, e2e_steps, world, e2e_ms)
    io_bytes = h0_host.numel() * h0_host.element_size()

    # ---------------- dense comparator (torch bf16 F.linear on W (.) M, same chain)
    dense = None
    if not args.no_dense:
        for _ in range(3):
            stack.dense_forward(h0)
        torch.cuda.synchronize()
        d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        nd = max(5, min(args.steps, 50))
        d0.record(s)
        for _ in range(nd):
            stack.dense_forward(h0)
        d1.record(s)
        torch.cuda.synchronize()
        dense_ms = d0.elapsed_time(d1) / nd
        stack_lin_ms = lin_ms / args.steps
        dense = {"dense_torch_ms_per_step": dense_ms, "speedup_linears_vs_dense": dense_ms / stack_lin_ms,
                 "speedup_step_vs_dense": dense_ms / (elapsed_ms / args.steps)}

    # ---------------- CPU oracle baseline (rank 0, N = 1)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        olayers = oracle_layers_from(layers)
        cores = os.cpu_count() or 1
        h_bits = inputs.bf16_bits(h0[:8192])
        rows = calibrate_rows(olayers, h_bits, cores, args.cpu_budget_s, 1)
        t0 = time.perf_counter()
        oracle_step(olayers, h_bits[:rows], cores)
        dt = time.perf_counter() - t0
        cpu = {"value": eff_flops_rows(olayers, rows) / dt / 1e12, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"first {rows} token rows through all 48 GEMMs (+ packing all 48 weights), one pass, "
                         f"fp64 C oracle on {cores} threads, {dt:.1f} s"}

    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": elapsed_max / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": WORKLOAD, "M": M_TOKENS, "block": BLOCK, "gemms": ngemm,
                   "sparsity": "per-GEMM U[0.30,0.70], antithetic layer pairs, mean 0.50",
                   "step": "pack all 48 weights + 48 chained block-sparse linears (fc1 with GELU)",
                   "launch": "one lpvit_bsr_linear_chain call (one launch)" if chain else "one call per linear",
                   "l2": "no flush: each step streams ~15 GB (> 129 MB L2)",
                   "parallelism": f"replicas x{world} (token batches per rank, no collective)"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "peak_source": f"{peak_src} bf16_tflops (burst, the dense bf16 cuBLAS rate)",
                     "kernel": ("lpvit::bsr_linear_chain_kernel" if chain
                                else "lpvit::bsr_linear_kernel<gelu, f32_out, deep>"),
                     "launches_timed": linear_launches,
                     "launch_timing": ("an event pair around every chain call" if chain else
                                       "an event pair around every linear") + ", in K steps run after the timed ones",
                     "frac_of_sustained_peak": achieved / peak_sustained,
                     "frac_of_nominal_peak": achieved / NOMINAL_BF16_TFLOPS,
                     "nominal_peak": "GB300 dense bf16 2250 TFLOP/s (datasheet, without 2:4 sparsity)"},
        "linear_ms_per_step": lin_ms / args.steps,
        "pack_ms_per_step": pack_ms / args.steps,
        "gaps_ms_per_step": (evpass_ms - pack_ms - lin_ms) / args.steps,
        "events_pass_ms_per_step": evpass_ms / args.steps,
        "hbm_gbs_linears": stack.algorithmic_bytes() * args.steps / (lin_ms / 1e3) / 1e9,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": io_bytes, "d2h_bytes_per_step": io_bytes,
                "steps": e2e_steps},
        "gpu_launches": args.steps * stack.launches_per_step(chain),
        "clocks": {"sm_mhz": clk["sm_mhz"], "sm_max_mhz": clk["sm_max_mhz"], "reasons": clk["reasons"],
                   "power_w_median": clk.get("power_w_median"), "samples": clk["samples"]},
        "cpu_baseline": cpu,
    }
    if dense:
        line.update(dense)
    print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_case(args, local):
    """One GEMM of the stack's shapes, pack + linear per step (for ncu and per-shape numbers)."""
    import torch
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    import paper_2407_02068_gb300 as lp
    from paper_2407_02068_gb300 import inputs
    k, n, b, sp, gelu, m = CASES[args.case]
    g = inputs.make_gemm(CONFIG_ID, 0, m, k, n, b, sp, device=dev)
    mask = g["mask"].to(dev).contiguous()
    w = lp.alloc_bsr(n, k, b, device=dev)
    Y = torch.empty(m, n, dtype=torch.bfloat16, device=dev)
    lp.pack_bsr_into(w, g["W"], mask)
    ws = lp.workspace_for(w, m)
    for _ in range(max(args.warmup, 1)):
        lp.pack_bsr_into(w, g["W"], mask)
        lp.bsr_linear(w, g["X"], g["bias"], gelu=gelu, out=Y, workspace=ws)
    lp.check(ws)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for e0, e1 in ev:
        lp.pack_bsr_into(w, g["W"], mask)
        e0.record()
        lp.bsr_linear(w, g["X"], g["bias"], gelu=gelu, out=Y, workspace=ws)
        e1.record()
    torch.cuda.synchronize()
    lp.check(ws)
    ms = sum(a.elapsed_time(b_) for a, b_ in ev) / len(ev)
    nnzb = int((g["mask"] != 0).sum())
    bn, bk = inputs.block_sides(b)
    flops = 2 * m * nnzb * bn * bk
    byts = 2 * m * k + 2 * m * n + 2 * nnzb * bn * bk + 4 * nnzb + 4 * (n // bn + 1) + 4 * n
    peaks, src = load_peaks()
    print(json.dumps({"case": args.case, "m": m, "k": k, "n": n, "b": b, "sparsity": sp, "gelu": gelu,
                      "linear_ms": ms, "eff_tflops": flops / ms / 1e9, "gbs": byts / ms / 1e6,
                      "frac_tensor_burst": flops / ms / 1e9 / float(peaks.get("bf16_tflops", 1900.0)),
                      "frac_hbm": byts / ms / 1e6 / float(peaks.get("hbm_gbs", 6800.0)), "peaks": src}),
          flush=True)


def _event_times(fn, before, min_ms, min_iters=50, max_iters=20000):
    """Per-call device times (ms) of fn() with CUDA events on the current stream; before() runs
    untimed ahead of each call (an L2 flush, or nothing). Iterates until min_ms of wall time and at
    least min_iters calls."""
    import torch
    evs = []
    t0 = time.perf_counter()
    while len(evs) < max_iters and (len(evs) < min_iters or (time.perf_counter() - t0) * 1e3 < min_ms):
        for _ in range(16):
            if before is not None:
                before()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            evs.append((e0, e1))
        torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in evs]


def run_config(args, local):
    """One line per GEMM of a named configuration: the block-sparse linear (bias, GELU on fc1, bf16
    output) timed with CUDA events after 10 warm-up calls, median and min over >= 50 calls and
    >= --min-ms of wall time, with a 2x-L2 buffer written before every call (cold L2, the primary
    number) and back to back (warm); at batch 1 also as a captured CUDA graph replay. Effective
    FLOPs F = 2 m nnzb bn bk; algorithmic bytes B = 2 m k_ref + 2 m n + 2 nnzb bn bk + 4 nnzb +
    4 (n/bn + 1) + 4 n (k_ref: the input columns of the block columns holding a kept block); the
    binding roof is max(F / P_bf16, B / BW) with the measured peaks. The pack (mask -> BSR + work
    list, an offline step per weight) and the dense torch bf16 linear on W (.) M are timed beside it."""
    import torch
    import torch.nn.functional as Fnn
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    import paper_2407_02068_gb300 as lp
    from paper_2407_02068_gb300 import inputs
    peaks, src = load_peaks()
    P = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    BW = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_buf = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)

    def flush():
        flush_buf.fill_(1.0)

    for (label, cfg, gi, m, k, n, b, sp, gelu, kind) in config_gemms(args.config):
        g = inputs.make_gemm(cfg, gi, m, k, n, b, sp, mask_kind=kind, device=dev)
        mask = g["mask"].to(dev).contiguous()
        bn, bk = inputs.block_sides(b)
        w = lp.alloc_bsr(n, k, b, device=dev)
        Y = torch.empty(m, n, dtype=torch.bfloat16, device=dev)
        lp.pack_bsr_into(w, g["W"], mask)
        ws = lp.workspace_for(w, m)
        call = lambda: lp.bsr_linear(w, g["X"], g["bias"], gelu=gelu, out=Y, workspace=ws)
        for _ in range(10):
            call()
        lp.check(ws)
        torch.cuda.synchronize()
        clk = ClockSampler(local)
        clk.start()
        time.sleep(0.3)
        cold = _event_times(call, flush, args.min_ms)
        warm = _event_times(call, None, args.min_ms)
        clocks = clk.stop()
        lp.check(ws)
        graph = None
        if m <= 256:
            try:
                cs = torch.cuda.Stream()
                cs.wait_stream(torch.cuda.current_stream())
                with torch.cuda.stream(cs):
                    for _ in range(3):
                        call()
                torch.cuda.current_stream().wait_stream(cs)
                torch.cuda.synchronize()
                gr = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gr):
                    call()
                gr.replay()
                torch.cuda.synchronize()
                lp.check(ws)
                gcold = _event_times(gr.replay, flush, args.min_ms)
                gwarm = _event_times(gr.replay, None, args.min_ms)
                lp.check(ws)
                graph = {"ms_median_cold": statistics.median(gcold), "ms_median_warm": statistics.median(gwarm),
                         "ms_min_warm": min(gwarm), "replays": len(gcold) + len(gwarm)}
            except Exception as e:  # capture refused: report why
                graph = {"error": f"{type(e).__name__}: {e}"[:200]}
        pack = _event_times(lambda: lp.pack_bsr_into(w, g["W"], mask), None, 50.0, min_iters=10)
        Wm = (g["W"].float() * mask.repeat_interleave(bn, 0).repeat_interleave(bk, 1).float()).to(torch.bfloat16)
        dense_fn = (lambda: Fnn.gelu(Fnn.linear(g["X"], Wm, g["bias"].to(torch.bfloat16)))) if gelu else \
            (lambda: Fnn.linear(g["X"], Wm, g["bias"].to(torch.bfloat16)))
        for _ in range(3):
            dense_fn()
        dense = _event_times(dense_fn, flush, 100.0, min_iters=20)
        Mh = g["mask"].numpy() != 0
        nnzb = int(Mh.sum())
        k_ref = bk * int(Mh.any(axis=0).sum())
        F = 2.0 * m * nnzb * bn * bk
        B = 2.0 * m * k_ref + 2.0 * m * n + 2.0 * nnzb * bn * bk + 4.0 * nnzb + 4.0 * (n // bn + 1) + 4.0 * n
        t = statistics.median(cold)
        t_roof = max(F / (P * 1e12), B / (BW * 1e9)) * 1e3
        bound = "hbm" if B / (BW * 1e9) >= F / (P * 1e12) else "tensor"
        achieved = (B / (t / 1e3) / 1e9) if bound == "hbm" else (F / (t / 1e3) / 1e12)
        line = {"metric": METRIC, "value": F / (t / 1e3) / 1e12, "unit": UNIT, "higher_is_better": True,
                "dtype": "bf16", "data": "synthetic",
                "config": {"workload": CONFIG_NAMES[args.config], "gemm": label, "config_id": cfg, "gemm_index": gi,
                           "m": m, "k": k, "n": n, "block": [bn, bk], "sparsity": sp, "mask": kind, "gelu": gelu,
                           "nnzb": nnzb, "l2": "2x L2 written before every timed call (cold); warm: back to back"},
                "ms_median": t, "ms_min": min(cold), "calls": len(cold),
                "warm_ms_median": statistics.median(warm), "warm_ms_min": min(warm),
                "eff_tflops": F / (t / 1e3) / 1e12, "gbs": B / (t / 1e3) / 1e9,
                "roofline": {"bound": bound, "achieved": achieved, "peak": BW if bound == "hbm" else P,
                             "unit": "GB/s" if bound == "hbm" else "TFLOP/s", "frac": achieved / (BW if bound == "hbm" else P),
                             "frac_of_roofline_time": t_roof / t, "peak_source": src,
                             "frac_tensor_burst": F / (t / 1e3) / 1e12 / P, "frac_hbm": B / (t / 1e3) / 1e9 / BW,
                             "frac_tensor_nominal": F / (t / 1e3) / 1e12 / NOMINAL_BF16_TFLOPS,
                             "frac_hbm_nominal": B / (t / 1e3) / 1e9 / NOMINAL_HBM_GBS},
                "algorithmic_bytes": B, "effective_flops": F,
                "graph": graph, "pack_ms_median": statistics.median(pack),
                "dense_torch_ms_median": statistics.median(dense),
                "speedup_vs_dense": statistics.median(dense) / t,
                "clocks": clocks}
        print(json.dumps(line), flush=True)
        del g, w, Y, ws, Wm
        torch.cuda.empty_cache()


def run_calibrate(args, local):
    """Cost-model calibration (Sec. 3.3, Eq. for P: p_m (M/B_m) ceil((1 - alpha) N K / (B_n B_k))):
    time each DeiT GEMM shape, with the block sizes of Table 2 (DeiT-B 32x32 and 64x32, DeiT-S
    16x16 and 16x32, printed output rows x input columns as Table 4's "BK x BN"; the transposed
    shapes are timed too), over a block-density sweep and fit, per shape, the least-squares line
    T = a + p * tiles * nnzb (tiles = ceil(M / 256), the kernel's token tile; nnzb = kept blocks).
    Prints one JSON line per shape with a, p (ns per block-tile), R^2 and the largest relative
    residual, and a final line with the fit over all shapes of each block size."""
    import numpy as np
    import torch
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    import paper_2407_02068_gb300 as lp
    from paper_2407_02068_gb300 import inputs
    shapes = []
    for blk in (32, (64, 32), (32, 64)):
        shapes += [("deit_b_fc1", 50432, 768, 3072, blk, True), ("deit_b_fc2", 50432, 3072, 768, blk, False),
                   ("deit_b_qkv", 50432, 768, 2304, blk, False), ("deit_b_proj", 50432, 768, 768, blk, False)]
    for blk in (16, (16, 32), (32, 16)):
        shapes += [("deit_s_fc1", 12608, 384, 1536, blk, True), ("deit_s_fc2", 12608, 1536, 384, blk, False)]
    densities = [1.0, 0.7, 0.5, 0.3, 0.2]
    reps = max(args.steps, 5)
    pooled = {}
    for si, (name, m, k, n, b, gelu) in enumerate(shapes):
        bn, bk = inputs.block_sides(b)
        X = inputs.activations(m, k, inputs.seed(6, si, "X"), dev)
        W = inputs.weight(n, k, inputs.seed(6, si, "W"), dev)
        bias = inputs.bias(n, inputs.seed(6, si, "bias"), dev)
        Y = torch.empty(m, n, dtype=torch.bfloat16, device=dev)
        xs, ts = [], []
        for d in densities:
            mask = inputs.uniform_mask(n, k, b, 1.0 - d, inputs.seed(6, si, "mask")).to(dev)
            w = lp.pack_bsr(W, mask, b, count=True)
            ws = lp.workspace_for(w, m)
            for _ in range(3):
                lp.bsr_linear(w, X, bias, gelu=gelu, out=Y, workspace=ws)
            times = []
            for _ in range(reps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                lp.bsr_linear(w, X, bias, gelu=gelu, out=Y, workspace=ws)
                e1.record()
                e1.synchronize()
                times.append(e0.elapsed_time(e1))
            lp.check(ws)
            xs.append(-(-m // 256) * w.nnzb)
            ts.append(float(np.median(times)) * 1e6)  # ns
        xs_a, ts_a = np.array(xs, dtype=np.float64), np.array(ts)
        A = np.stack([np.ones_like(xs_a), xs_a], axis=1)
        (a, p_), *_ = np.linalg.lstsq(A, ts_a, rcond=None)
        pred = a + p_ * xs_a
        r2 = 1 - np.sum((ts_a - pred) ** 2) / np.sum((ts_a - ts_a.mean()) ** 2)
        print(json.dumps({"shape": name, "m": m, "k": k, "n": n, "block": f"{bn}x{bk}", "gelu": gelu,
                          "densities": densities,
                          "block_tiles": xs, "median_ns": ts, "a_ns": a, "p_ns_per_block_tile": p_, "r2": r2,
                          "max_rel_residual": float(np.max(np.abs(ts_a - pred) / ts_a))}), flush=True)
        pooled.setdefault(f"{bn}x{bk}", []).extend(zip(xs, ts))
    for b, pts in pooled.items():
        xs_a = np.array([x for x, _ in pts], dtype=np.float64)
        ts_a = np.array([t for _, t in pts])
        A = np.stack([np.ones_like(xs_a), xs_a], axis=1)
        (a, p_), *_ = np.linalg.lstsq(A, ts_a, rcond=None)
        pred = a + p_ * xs_a
        r2 = 1 - np.sum((ts_a - pred) ** 2) / np.sum((ts_a - ts_a.mean()) ** 2)
        print(json.dumps({"pooled_over_shapes_block": b, "a_ns": a, "p_ns_per_block_tile": p_, "r2": r2,
                          "max_rel_residual": float(np.max(np.abs(ts_a - pred) / ts_a))}), flush=True)


def run_alloc(args, local):
    """Pruning-ratio allocation (Sec. 3.4-3.5) for the 12-layer DeiT-B linear stack, 32x32 blocks:
    the distortion curve of each of the 48 weights from N seeded per-sample gradients (20 ratio
    steps, kappa 1e-3; the weights are independent and go round-robin to --alloc-streams CUDA streams,
    each with its own workspace; every weight's gradients are generated on the device before the
    timed region), then the host lambda search at a 50% FLOPs target. One JSON line:
    throughput in GB/s of algorithmic bytes (the gradients and the weight read once), against the
    measured HBM copy bandwidth; the oracle is timed on one qkv weight."""
    import torch
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    import paper_2407_02068_gb300 as lp
    from paper_2407_02068_gb300 import inputs
    N, steps, kappa, b, m = args.alloc_samples, 20, 1e-3, 32, M_TOKENS
    shapes = [(gi, k, n) for l in range(12) for gi, (_, k, n, _) in
              ((4 * l + t, g) for t, g in enumerate(inputs.deit_gemms(inputs.DEIT_B)))]
    Ws = [inputs.weight(n, k, inputs.seed(8, gi, "W"), dev) for gi, k, n in shapes]
    gen = torch.Generator(device=dev)
    ws_bytes = max(lp._lib.lpvit_delta_curve_workspace_bytes(N, n, k, b, b, steps) for _, k, n in shapes)
    ns = max(1, args.alloc_streams)
    wss = [torch.empty(ws_bytes, dtype=torch.uint8, device=dev) for _ in range(ns)]

    def grads(gi, k, n):
        gen.manual_seed(inputs.seed(8, gi, "X"))
        Gv = torch.empty(N, n, k, dtype=torch.float32, device=dev)
        Gv.normal_(0.0, 1e-2, generator=gen)
        return Gv

    Gs = [grads(gi, k, n) for gi, k, n in shapes]  # all resident (N x 85 M floats) before timing
    streams = [torch.cuda.Stream(dev) for _ in range(ns)]
    main = torch.cuda.current_stream(dev)

    def one_pass():
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(main)
        for st in streams:
            st.wait_event(e0)
        ds = []
        for i, ((gi, k, n), W) in enumerate(zip(shapes, Ws)):
            st = streams[i % ns]
            with torch.cuda.stream(st):
                ds.append(lp.delta_curve(W, Gs[i], b, steps, kappa, workspace=wss[i % ns], stream=st))
        for st in streams:
            ev = torch.cuda.Event()
            ev.record(st)
            main.wait_event(ev)
        e1.record(main)
        e1.synchronize()
        return e0.elapsed_time(e1), ds

    one_pass()  # warm-up
    torch.cuda.synchronize()
    clk = ClockSampler(local)
    clk.start()
    total_ms, ds = one_pass()
    clocks = clk.stop()
    curves = [d.cpu().numpy() for d in ds]
    algo = sum(4 * N * n * k + 2 * n * k for _, k, n in shapes)
    F = [float(m * n * k) for _, k, n in shapes]
    c = [float(m * n * k) / (b * b) for _, k, n in shapes]
    t0 = time.perf_counter()
    ks, lam, ratio = lp.lambda_search(curves, steps, F, c, 1e-12, 0.5)
    search_ms = (time.perf_counter() - t0) * 1e3
    peaks, src = load_peaks()
    achieved = algo / (total_ms / 1e3) / 1e9
    line = {"metric": "pruning-ratio allocation: distortion-curve throughput (per-sample gradients + weights)",
            "value": achieved, "unit": "GB/s", "n_gpus": 1, "higher_is_better": True, "dtype": "f64",
            "data": "synthetic", "config": {"workload": "deit_b_12layer_allocation", "weights": 48, "block": b,
                                            "samples": N, "ratio_steps": steps, "kappa": kappa, "streams": ns,
                                            "flops_target": 0.5, "beta": 1e-12},
            "ms_total": total_ms, "lambda_search_ms": search_ms, "allocated_k": ks, "flops_remained": ratio,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": float(peaks.get("hbm_gbs", 6800.0)),
                         "unit": "GB/s", "frac": achieved / float(peaks.get("hbm_gbs", 6800.0)), "traffic": None,
                         "peak_source": src + " hbm_gbs (STREAM-style copy)"},
            "gpu_launches": 8 * len(shapes), "clocks": clocks}
    if not args.no_cpu_baseline:
        import oracle.alloc as oalloc
        gi, k, n = shapes[0]
        Wb = inputs.bf16_bits(Ws[0])
        Gh = Gs[0].cpu().numpy()
        t0 = time.perf_counter()
        oalloc.delta_curve(Wb, Gh, b, steps, kappa)
        cpu_s = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": (4 * N * n * k + 2 * n * k) / cpu_s / 1e9, "unit": "GB/s",
                                "cores": os.cpu_count(), "kind": "oracle",
                                "sample": f"one qkv weight ({n}x{k}), {N} samples, {steps + 1} ratios, numpy fp64 "
                                          f"with its default BLAS threading, {cpu_s:.1f} s"}
    print(json.dumps(line), flush=True)


def run_encoder(args, local):
    """End-to-end pre-norm encoder forward (the pruned ViTs of Sec. 4): DeiT-B (12 layers, 768 wide,
    12 heads) or DeiT-S (12 layers, 384 wide, 6 heads), 32x32 blocks with the stack's per-GEMM
    sparsities (U[0.30, 0.70], mean 50%), seeded random weights, masks, biases and LayerNorm
    parameters, 197-token images. Times the library's forward (every step in liblpvit.so: 2
    add+LayerNorms, 4 block-sparse linears and attention per layer, a final LayerNorm) and the same
    model on torch's dense bf16 operations, with CUDA events; the speedup over dense is the measure
    the paper reports end to end on its A100. e2e adds the host->device copy of the images and the
    device->host copy of the output every step."""
    import torch
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2407_02068_gb300 import inputs
    from paper_2407_02068_gb300.encoder import SparseEncoder
    model = inputs.DEIT_B if args.encoder == "deit_b" else inputs.DEIT_S
    D, hidden, heads, T, b = model["dim"], model["hidden"], model["dim"] // 64, 197, 32
    config = 9
    layers, final = inputs.deit_encoder_params(model, b, config, 12, dev)
    enc = SparseEncoder(layers, final, heads, T, b)
    M = args.images * T
    x = inputs.activations(M, D, inputs.seed(config, 0, "X"), dev)
    steps, warm = max(args.steps // 20, 5), max(args.warmup, 3)

    def timed(fn):
        for _ in range(warm):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(steps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / steps

    clk = ClockSampler(local)
    clk.start()
    ms_sparse = timed(lambda: enc.forward(x))
    clocks = clk.stop()
    ms_dense = timed(lambda: enc.dense_forward(x))
    # end to end: pinned host images in, output back, every step, on a copy stream overlapping the
    # forwards: the input double-buffered on the device (step k+1's copy runs during step k), the
    # output staged by a device copy the step pays for and copied out during the next step
    xh = x.cpu().pin_memory()
    yh = torch.empty((M, D), dtype=torch.bfloat16).pin_memory()
    xd = [torch.empty_like(x), torch.empty_like(x)]
    stage = torch.empty((M, D), dtype=torch.bfloat16, device=dev)
    s = torch.cuda.current_stream()
    cs = torch.cuda.Stream(device=dev)
    in_ready = [torch.cuda.Event(), torch.cuda.Event()]
    in_free = [torch.cuda.Event(), torch.cuda.Event()]
    out_ready, out_done = torch.cuda.Event(), torch.cuda.Event()

    def e2e_run(n):
        cs.wait_stream(s)
        with torch.cuda.stream(cs):
            xd[0].copy_(xh, non_blocking=True)
            in_ready[0].record(cs)
            out_done.record(cs)
        for k in range(n):
            s.wait_event(in_ready[k % 2])
            y = enc.forward(xd[k % 2])
            in_free[k % 2].record(s)
            if k + 1 < n:
                nb = (k + 1) % 2
                if k >= 1:
                    cs.wait_event(in_free[nb])  # forward k - 1 has finished with this buffer
                with torch.cuda.stream(cs):
                    xd[nb].copy_(xh, non_blocking=True)
                    in_ready[nb].record(cs)
            s.wait_event(out_done)  # the stage's previous result is in host memory
            stage.copy_(y, non_blocking=True)
            out_ready.record(s)
            cs.wait_event(out_ready)
            with torch.cuda.stream(cs):
                yh.copy_(stage, non_blocking=True)
                out_done.record(cs)
        s.wait_event(out_done)

    e2e_run(warm)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s)
    e2e_run(steps)
    e1.record(s)
    torch.cuda.synchronize()
    ms_e2e = e0.elapsed_time(e1) / steps
    dense_flops = sum(2 * M * k * n for l in range(12) for (_, k, n, _) in inputs.deit_gemms(model))
    eff_flops = sum(2 * M * int((L[name][1] != 0).sum()) * b * b for L in layers for name in ("qkv", "proj", "fc1", "fc2"))
    line = {"metric": f"end-to-end {args.encoder} encoder forward throughput", "value": args.images / (ms_sparse / 1e3),
            "unit": "images/s", "n_gpus": 1, "steps": steps, "warmup": warm, "ms_per_step": ms_sparse,
            "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": f"{args.encoder}_12layer_encoder_batch{args.images}", "images": args.images,
                       "tokens": T, "block": b, "sparsity": "per-GEMM U[0.30,0.70], antithetic layer pairs, mean 0.50",
                       "flops_remained_linears": eff_flops / dense_flops},
            "dense_torch_ms_per_step": ms_dense, "speedup_vs_dense": ms_dense / ms_sparse,
            "e2e": {"value": args.images / (ms_e2e / 1e3), "unit": "images/s", "h2d_bytes_per_step": 2 * M * D,
                    "d2h_bytes_per_step": 2 * M * D},
            "gpu_launches": steps * enc.launches(), "clocks": clocks}
    if not args.no_cpu_baseline:
        import numpy as np
        import oracle
        from oracle import encoder as oenc
        ol = []
        for L in layers:
            d = {"ln1": tuple(v.cpu().double().numpy() for v in L["ln1"]),
                 "ln2": tuple(v.cpu().double().numpy() for v in L["ln2"])}
            for name in ("qkv", "proj", "fc1", "fc2"):
                W, Mk, bias = L[name]
                d[name] = (inputs.bf16_bits(W), Mk.cpu().numpy(), bias.cpu().numpy(), b)
            ol.append(d)
        of = tuple(v.cpu().double().numpy() for v in final)
        t0 = time.perf_counter()
        oenc.encoder_forward(inputs.bf16_bits(x[:T]), ol, of, T, heads)
        cpu_s = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": 1.0 / cpu_s, "unit": "images/s", "cores": os.cpu_count(), "kind": "oracle",
                                "sample": f"one image through the 12-layer encoder, fp64 C/numpy oracle, {cpu_s:.1f} s"}
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, world, rank)
        return
    if args.calibrate:
        run_calibrate(args, local)
        return
    if args.alloc:
        run_alloc(args, local)
        return
    if args.encoder:
        run_encoder(args, local)
        return
    if args.config is not None:
        run_config(args, local)
        return
    if args.case != "stack":
        run_case(args, local)
        return
    run_gpu(args, world, rank, local)


if __name__ == "__main__":
    main()
