#!/usr/bin/env python
"""Benchmark of the MXINT mixed-precision linear layer (MXSens) on GB300.

Default workload (LLaMA-3-8B-shaped decode): for M in {1, 4, 16} tokens, the
seven projections (q, k, v, o: 4096x4096 / 4096x1024; gate, up: 4096x14336;
down: 14336x4096) of all 32 decoder layers; width map 85/10/5 % (4/6/8 bits)
per projection, weights N(0, 0.02), activations N(0, 1) with 1 % outlier
columns x30.  One step = for every (M, layer, projection): quantize the
activations (A1) and run the MXINT GEMM (A4); weights are packed once (A2).
The step is captured in a CUDA graph and replayed.  The 4.2 GB of packed
weights a step streams is far larger than L2, so no flush is needed.

Metric: GB/s of algorithmic traffic (packed weights + bf16 activations read +
fp32 outputs written) per second, whole job; TOPS (2*M*N*K per second) is
reported beside it.

--impl reference times the CPU oracle (the paper publishes no kernel to run)
on a bounded sample of the same workload, on the host cores.
"""
from __future__ import annotations

import argparse
import math
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_17733_gb300 import inputs as I  # noqa: E402

DECODE_MS = (1, 4, 16)
MAP = (0.85, 0.10, 0.05)
W_SIGMA = 0.02
OUTLIER_FRAC, OUTLIER_SCALE = 0.01, 30.0
SEED = 2607
SAMPLE_ROWS = 2048


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--layers", type=int, default=None,
                    help="decoder layers per step (default 32 for decode, 8 for prefill)")
    ap.add_argument("--workload", default="llama3-8b-decode",
                    choices=["llama3-8b-decode", "llama3-8b-prefill", "llama3-8b-calibration",
                             "llama3-8b-decode-attention"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--path", default="grouped", choices=["planes", "fused", "codes", "grouped"],
                    help="decode activation path: quantize all projections to MMA planes, then the GEMMs "
                         "(planes); mxs_linear_decode per projection, the GEMM a programmatic dependent of "
                         "its quantizer (fused); quantize to packed codes, GEMM over the codes (codes); as fused, "
                         "but the projections that share an input in a decoder layer (q/k/v, gate/up) in one "
                         "grouped GEMM launch (grouped)")
    ap.add_argument("--eager", action="store_true",
                    help="launch the step's kernels directly (no CUDA graph, no events): for ncu runs")
    return ap.parse_args()


# --------------------------------------------------------------- helpers
def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def profile_traffic(kernel_file: str, profile_md: str):
    """DRAM bytes per launch recorded in a committed ncu summary, if it was taken
    on the current source of the kernel (sha256 of the .cu file)."""
    import hashlib
    try:
        src = open(os.path.join(ROOT, "paper_2607_17733_gb300", "csrc", kernel_file), "rb").read()
        text = open(os.path.join(ROOT, "profiles", profile_md)).read()
    except OSError:
        return None
    sha = hashlib.sha256(src).hexdigest()[:16]
    for line in text.splitlines():
        if line.startswith("traffic_bytes_per_launch:"):
            parts = line.split()
            # traffic_bytes_per_launch: <bytes> kernel_sha: <sha>
            if len(parts) >= 4 and parts[3] == sha:
                return float(parts[1])
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.proc = None
        self.lines = []
        self.gpu_id = gpu_id

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50"]
        if self.gpu_id:
            cmd += ["-i", self.gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.12)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("gloo", rank=rank, world_size=ws)  # harness barriers / max only
    return ws, rank, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def allreduce_max(v: float, ws: int) -> float:
    if ws == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------- CPU oracle sample
_SAMPLE = None


def _oracle_jobs(seed_rank: int = 0):
    """Layer 0 of the workload for the oracle, the first min(N, 2048) output
    rows of every projection: weights quantized once (offline packing is not
    timed), activations for M = 1, 4, 16."""
    global _SAMPLE
    if _SAMPLE is None:
        from oracle import mxo
        jobs = []
        for pi, (name, K, N) in enumerate(I.LLAMA3_8B):
            g = I.rng(SEED, seed_rank, 0, pi)
            bits = I.width_map(K // 32, *MAP, g)
            N = min(N, SAMPLE_ROWS)
            w = I.normal_bf16((N, K), W_SIGMA, g)
            w_s, w_c = mxo.quantize_bf16(w, bits)
            del w
            for M in DECODE_MS:
                x = I.activations_bf16(M, bits, I.rng(SEED, seed_rank, 1, pi, M), OUTLIER_FRAC,
                                       outlier_scale=OUTLIER_SCALE)
                jobs.append((bits, x, w_s, w_c, K, N, M))
        _SAMPLE = jobs
    return _SAMPLE


def oracle_sample(min_seconds: float = 10.0):
    """Time the oracle on a bounded sample of the step: the quantization and
    exact GEMM of layer 0's seven projections at M = 1, 4, 16 (the first
    min(N, 2048) output columns of each), passes
    repeated until min_seconds have elapsed (at least one).  Returns (GB/s of
    the same algorithmic traffic as the GPU step, seconds, threads, text)."""
    from oracle import mxo
    jobs = _oracle_jobs()
    t0 = time.perf_counter()
    nbytes = 0
    passes = 0
    while True:
        for bits, x, w_s, w_c, K, N, M in jobs:
            a_s, a_c = mxo.quantize_bf16(x, bits)
            mxo.gemm(bits, a_c, a_s, w_c, w_s)
            n4 = int(np.sum(bits == 4))
            nbytes += N * (16 * n4 + 32 * (bits.size - n4) + bits.size) + M * K * 2 + M * N * 4
        passes += 1
        if time.perf_counter() - t0 >= min_seconds:
            break
    dt = time.perf_counter() - t0
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    desc = (f"layer 0 (q/k/v/o/gate/up/down, first min(N,{SAMPLE_ROWS}) output columns) at M=1,4,16, "
            f"{passes} pass(es): oracle "
            f"activation quantization + exact GEMM, OpenMP over output rows")
    return nbytes / dt / 1e9, dt, threads, desc


def run_reference(args):
    ws, rank, _ = dist_setup()
    if rank != 0:
        return
    for _ in range(args.warmup):
        oracle_sample(min_seconds=0.0)
    vals, secs = [], []
    for _ in range(args.steps):
        v, dt, threads, desc = oracle_sample(min_seconds=0.0)
        vals.append(v)
        secs.append(dt)
    value = statistics.median(vals)
    line = {
        "impl": "reference", "metric": "mxint_decode_gemm_gbps", "value": value, "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * statistics.median(secs), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int64+f64", "data": "synthetic",
        "config": {"workload": "llama3-8b-decode (sample)", "layers": 1, "M": list(DECODE_MS)},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": threads, "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------- GPU arm
def run_ours(args):
    import torch

    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_17733_gb300 import build as B
    from paper_2607_17733_gb300 import mxs
    from paper_2607_17733_gb300.runtime import MxLinear
    if not os.path.exists(mxs.LIB_PATH):
        B.build()
    mxs.lib()

    L = args.layers
    # ---- weights: drawn on the GPU (seeded per layer/projection), packed once
    layers = []
    gen = torch.Generator(device=dev)
    for l in range(L):
        projs = []
        for pi, (name, K, N) in enumerate(I.LLAMA3_8B):
            bits = I.width_map(K // 32, *MAP, I.rng(SEED, rank, l, pi))
            gen.manual_seed(SEED * 1_000_003 + rank * 10_007 + l * 101 + pi)
            w = (torch.randn((N, K), generator=gen, device=dev, dtype=torch.float32) * W_SIGMA).to(torch.bfloat16)
            projs.append(MxLinear(w, bits))
            del w
        layers.append(projs)
    torch.cuda.synchronize()

    # ---- inputs: one contiguous pinned host block and one device block per step
    items = []  # (M, lin, x_dev, bufs)
    x_sizes = []
    for M in DECODE_MS:
        for l in range(L):
            for pi, lin in enumerate(layers[l]):
                x_sizes.append(M * lin.K)
    x_host = torch.empty(sum(x_sizes), dtype=torch.bfloat16, pin_memory=True)
    x_dev = torch.empty_like(x_host, device=dev)
    y_sizes = []
    off = 0
    xi = 0
    for M in DECODE_MS:
        for l in range(L):
            for pi, lin in enumerate(layers[l]):
                xb = I.activations_bf16(M, lin.bits, I.rng(SEED, rank, 2, M, l, pi), OUTLIER_FRAC,
                                        outlier_scale=OUTLIER_SCALE)
                n = M * lin.K
                x_host[off:off + n].copy_(torch.from_numpy(xb.view(np.int16).ravel()).view(torch.bfloat16))
                bufs = lin.buffers(M, dev)
                items.append((M, lin, x_dev[off:off + n].view(M, lin.K), bufs))
                y_sizes.append(M * lin.N)
                off += n
                xi += 1
    y_dev = torch.empty(sum(y_sizes), dtype=torch.float32, device=dev)
    y_host = torch.empty_like(y_dev, device="cpu", pin_memory=True)
    off = 0
    for (M, lin, x, bufs), n in zip(items, y_sizes):
        bufs["y"] = y_dev[off:off + n].view(M, lin.N)
        off += n
    x_dev.copy_(x_host)
    torch.cuda.synchronize()

    # ---- algorithmic work per step
    step_bytes = sum(lin.weight_bytes + M * lin.K * 2 + M * lin.N * 4 for M, lin, _, _ in items)
    step_ops = sum(2 * M * lin.N * lin.K for M, lin, _, _ in items)
    if args.path == "codes":  # the GEMM reads the packed codes the quantizer wrote
        gemm_bytes = sum(lin.weight_bytes + M * (mxs.act_row_bytes(lin.K, lin.bits) + lin.K // 32) + M * lin.N * 4
                         for M, lin, _, _ in items)
    elif args.path == "planes":  # the GEMM reads the activations' MMA planes (digits + scale tiles)
        gemm_bytes = sum(lin.weight_bytes + mxs.act_planes_bytes(M, lin.K, lin.bits) + M * lin.N * 4
                         for M, lin, _, _ in items)
    else:  # the timed segment is quantize + GEMM: bf16 activations in, y out
        gemm_bytes = step_bytes
    launches_per_step = 2 * len(items)
    STAGES = [[0, 1, 2], [3], [4, 5], [6]]  # q k v | o | gate up | down: the projections of a stage share an input
    if args.path == "grouped":  # per stage one quantizer launch and one GEMM launch
        launches_per_step = 2 * len(items) // 7 * len(STAGES)

    # ---- the step as one CUDA graph.  Inputs are independent synthetic draws, so
    # for each M the graph runs all activation quantizations, then all GEMMs;
    # on one stream every kernel waits for the previous one either way.  Two
    # event nodes per M bracket the GEMM segment: the dominant kernel's time
    # is read from them for every timed step, at 6 event nodes per step.
    capture_stream = torch.cuda.Stream(device=dev)
    groups = [[it for it in items if it[0] == M] for M in DECODE_MS]

    def make_step(events=None):
        def fn():
            for gi, grp in enumerate(groups):
                if args.path not in ("fused", "grouped"):
                    for M, lin, x, bufs in grp:
                        if args.path == "codes":
                            lin.quantize(x, bufs)
                        else:
                            mxs.quantize_act(x, lin.bits, rounding=lin.rounding, planes=bufs["planes"],
                                             want_codes=False, want_planes=True)
                if events is not None:
                    events[gi][0].record()
                if args.path == "grouped":
                    for base in range(0, len(grp), 7):
                        for stage in STAGES:
                            its = [grp[base + i] for i in stage]
                            if len(its) == 1:
                                M, lin, x, bufs = its[0]
                                lin.fused(x, bufs["y"], bufs["planes"])
                            else:
                                mxs.linear_decode_group([(x, lin.bits, lin.packed, lin.N, bufs["y"], bufs["planes"])
                                                         for M, lin, x, bufs in its])
                for M, lin, x, bufs in (grp if args.path != "grouped" else []):
                    if args.path == "codes":
                        lin.matmul(bufs)
                    elif args.path == "planes":
                        mxs.gemm_decode(None, None, lin.bits, lin.packed, lin.N, y=bufs["y"], planes=bufs["planes"],
                                        M=M)
                    else:
                        lin.fused(x, bufs["y"], bufs["planes"])
                if events is not None:
                    events[gi][1].record()
        return fn

    def capture(fn):
        capture_stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(capture_stream):
            fn()
        capture_stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=capture_stream):
            fn()
        torch.cuda.synchronize()
        return g

    if args.eager:  # profiling mode: plain launches, nothing else timed or printed
        fn = make_step()
        for _ in range(args.warmup + args.steps):
            fn()
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"eager_steps": args.steps, "launches_per_step": launches_per_step}), flush=True)
        return

    plain = capture(make_step())
    try:
        ev_sets = [[(torch.cuda.Event(enable_timing=True, external=True),
                     torch.cuda.Event(enable_timing=True, external=True)) for _ in groups]
                   for _ in range(args.steps)]
        timed = [capture(make_step(evs)) for evs in ev_sets]
    except TypeError:  # torch without external events: time the plain graph only
        ev_sets, timed = None, [plain] * args.steps

    for _ in range(args.warmup):
        plain.replay()
    torch.cuda.synchronize()

    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid).replace("GPU-", "")
    except Exception:
        pass
    sampler = ClockSampler(gpu_id)

    # ---- timed region (device time, max over ranks)
    barrier(ws)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.1)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for k in range(args.steps):
        timed[k].replay()
    t1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    barrier(ws)
    ms = t0.elapsed_time(t1) / args.steps
    ms = allreduce_max(ms, ws)
    value = ws * step_bytes / (ms * 1e-3) / 1e9
    tops = ws * step_ops / (ms * 1e-3) / 1e12

    # ---- the dominant kernel (decode GEMM): per-launch durations from the graphs' events
    pk = peaks()
    roofline = None
    if ev_sets is not None:
        gemm_ms = sum(s.elapsed_time(e) for evs in ev_sets for s, e in evs) / len(ev_sets)  # per step
        achieved = gemm_bytes / (gemm_ms * 1e-3) / 1e9
        traffic = profile_traffic("gemm_decode.cu", "gemm_decode_llama3_8b_decode.md")
        roofline = {"kernel": "gemm_decode_kernel" + (" + quantize_act_kernel (PDL chain)"
                                                      if args.path in ("fused", "grouped") else f" ({args.path} path)"),
                    "bound": "hbm", "achieved": achieved,
                    "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": achieved / pk["hbm_gbs"],
                    "peak_source": pk["source"], "traffic": traffic,
                    "bytes_per_step": gemm_bytes, "gemm_ms_per_step": gemm_ms,
                    "gemm_launches_per_step": len(items) // 7 * len(STAGES) if args.path == "grouped" else len(items),
                    "share_of_step": gemm_ms / ms}

    # ---- end to end through the public API with host buffers
    barrier(ws)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e2e_steps = max(1, min(args.steps, 50))
    e0.record()
    for _ in range(e2e_steps):
        x_dev.copy_(x_host, non_blocking=True)
        plain.replay()
        y_host.copy_(y_dev, non_blocking=True)
    e1.record()
    torch.cuda.synchronize()
    e2e_ms = allreduce_max(e0.elapsed_time(e1) / e2e_steps, ws)
    e2e = {"value": ws * step_bytes / (e2e_ms * 1e-3) / 1e9, "unit": "GB/s",
           "h2d_bytes_per_step": x_host.numel() * 2, "d2h_bytes_per_step": y_host.numel() * 4,
           "ms_per_step": e2e_ms}

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, dt, threads, desc = oracle_sample()
        cpu = {"value": v, "unit": "GB/s", "cores": threads, "kind": "oracle", "sample": desc, "seconds": dt}

    if rank == 0:
        line = {
            "metric": "mxint_decode_gemm_gbps", "value": value, "unit": "GB/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int8+f32",
            "data": "synthetic (seeded; weights N(0,0.02), activations N(0,1) with 1% outlier columns x30)",
            "config": {"workload": "llama3-8b-decode", "M": list(DECODE_MS), "layers": L,
                       "path": {"planes": "quantize to MMA planes, then GEMM over the planes (TMA)",
                                "fused": "mxs_linear_decode: quantize + GEMM chained by programmatic dependent launch",
                                "grouped": "mxs_linear_decode_group for q/k/v and gate/up (one GEMM launch per "
                                           "group, after one quantizer launch for the group), mxs_linear_decode for o, down",
                                "codes": "quantize to packed codes, GEMM over the codes"}[args.path],
                       "projections": [p[0] for p in I.LLAMA3_8B], "map_4_6_8": list(MAP),
                       "parallelism": f"replicas x{ws}", "l2": "inputs larger than L2 (packed weights "
                       f"{sum(lin.weight_bytes for p in layers for lin in p) / 1e9:.2f} GB per step)"},
            "tops": tops,
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches_per_step * args.steps,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)


def run_prefill(args):
    """LLaMA-3-8B-shaped prefill: M = 2048 tokens through q/k/v/o/gate/up/down of
    `layers` layers, map 80/15/5, activations N(0,1) with Student-t(3) outlier
    channels on 0.5 % of K.  Per stage of a layer (q/k/v, o, gate/up, down: the
    projections of a stage read one hidden state): one quantizer launch to MMA
    planes (A1) for its projections, then their tcgen05 GEMMs (A3).  Metric:
    effective TOPS = 2*M*N*K / s, whole job."""
    import torch

    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_17733_gb300 import build as B
    from paper_2607_17733_gb300 import mxs
    from paper_2607_17733_gb300.runtime import MxLinear
    if not os.path.exists(mxs.LIB_PATH):
        B.build()
    mxs.lib()
    M = 2048
    L = args.layers or 8
    gen = torch.Generator(device=dev)
    items = []
    for l in range(L):
        for pi, (name, K, N) in enumerate(I.LLAMA3_8B):
            bits = I.width_map(K // 32, 0.80, 0.15, 0.05, I.rng(SEED, rank, 3, l, pi))
            gen.manual_seed(SEED * 7 + rank * 10_007 + l * 101 + pi)
            w = (torch.randn((N, K), generator=gen, device=dev, dtype=torch.float32) * W_SIGMA).to(torch.bfloat16)
            lin = MxLinear(w, bits, with_planes=True)
            del w
            items.append((lin, bits))
    planes, ys = [], []
    for idx, (lin, bits) in enumerate(items):
        # N(0,1) activations, 0.5 % of K channels (inside 8-bit blocks) redrawn from
        # a Student-t(3) = Z / sqrt(chi2_3 / 3); drawn on the GPU from a seeded stream
        gen.manual_seed(SEED * 13 + rank * 10_007 + idx)
        x = torch.randn((M, lin.K), generator=gen, device=dev, dtype=torch.float32)
        cols = torch.from_numpy(I.outlier_columns(bits, int(np.floor(0.005 * lin.K + 0.5)),
                                                  I.rng(SEED, rank, 6, idx))).to(dev)
        z = torch.randn((M, cols.numel(), 4), generator=gen, device=dev, dtype=torch.float32)
        x[:, cols] = z[..., 0] / torch.sqrt((z[..., 1:] ** 2).sum(-1) / 3.0)
        x = x.to(torch.bfloat16)
        planes.append((x, torch.empty(mxs.act_planes_bytes(M, lin.K, bits), dtype=torch.uint8, device=dev)))
        ys.append(torch.empty((M, lin.N), dtype=torch.float32, device=dev))
    torch.cuda.synchronize()
    step_ops = sum(2 * M * lin.N * lin.K for lin, _ in items)

    # the projections of a stage read one hidden state (q/k/v; gate/up): their
    # activations are quantized by one launch, then their GEMMs run
    PSTAGES = [[0, 1, 2], [3], [4, 5], [6]]
    n_launch = len(items) + len(items) // 7 * len(PSTAGES)

    def fn(events=None):
        for base in range(0, len(items), 7):
            for stage in PSTAGES:
                idxs = [base + i for i in stage]
                if len(idxs) == 1:
                    x, pl = planes[idxs[0]]
                    mxs.quantize_act(x, items[idxs[0]][1], planes=pl, want_codes=False)
                else:
                    mxs.quantize_act_group([(planes[i][0], items[i][1], planes[i][1]) for i in idxs])
                for idx in idxs:
                    lin, bits = items[idx]
                    if events is not None:
                        events[idx][0].record()
                    mxs.gemm_prefill(planes[idx][1], bits, lin.packed, M, lin.N, y=ys[idx])
                    if events is not None:
                        events[idx][1].record()

    if args.eager:
        for _ in range(args.warmup + args.steps):
            fn()
        torch.cuda.synchronize()
        print(json.dumps({"eager_steps": args.steps, "launches_per_step": n_launch}), flush=True)
        return
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in items]
           for _ in range(args.steps)]
    sampler = ClockSampler(None)
    barrier(ws)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.1)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for k in range(args.steps):
        fn(evs[k])
    t1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = allreduce_max(t0.elapsed_time(t1) / args.steps, ws)
    gemm_ms = sum(s.elapsed_time(e) for ev in evs for s, e in ev) / args.steps
    pk = peaks()
    fp8_peak = 2.0 * pk["bf16_tflops"]
    achieved = step_ops / (gemm_ms * 1e-3) / 1e12
    value = ws * step_ops / (ms * 1e-3) / 1e12
    if rank == 0:
        print(json.dumps({
            "metric": "mxint_prefill_gemm_tops", "value": value, "unit": "TOPS", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "e4m3 (4-bit blocks) + bf16 (6/8-bit blocks), f32 accumulation",
            "data": "synthetic (seeded; W N(0,0.02), A N(0,1) with Student-t(3) outlier channels on 0.5% of K)",
            "config": {"workload": "llama3-8b-prefill", "M": M, "layers": L, "map_4_6_8": [0.8, 0.15, 0.05],
                       "l2": "inputs larger than L2"},
            "roofline": {"kernel": "gemm_prefill_kernel", "bound": "tensor", "achieved": achieved,
                         "peak": fp8_peak, "unit": "TFLOP/s", "frac": achieved / fp8_peak,
                         "peak_source": pk["source"] + " bf16 x 2 (fp8/bf16 nominal ratio)",
                         "traffic": profile_traffic("gemm_prefill.cu", "gemm_prefill_llama3_8b_prefill.md"),
                         "gemm_ms_per_step": gemm_ms, "share_of_step": gemm_ms / ms},
            "gpu_launches": n_launch * args.steps, "clocks": clocks}), flush=True)


CALIB_SEQ, CALIB_BATCH = 2048, 8  # a calibration sample is a 2048-token sequence; 8 samples per call


def run_calibration(args):
    """Alg. 1 over calibration activations (offline allocation): one step adds
    a batch of 8 calibration samples of 2048 tokens (16384 rows) into the
    column sensitivities of the four distinct linear-layer inputs of `layers`
    LLaMA-3-8B-shaped layers (default 8): the
    attention input (shared by q/k/v), the output projection's, the MLP input
    (shared by gate/up) and the down projection's (K = 4096, 4096, 4096,
    14336).  Activations N(0,1) with 1 % of the columns x50 (systematic
    outlier channels), drawn on the GPU from a seeded stream: synthetic
    stand-ins for the paper's C4 calibration samples.  Metric: GB/s of bf16
    activations reduced (HBM-bound).  Alg. 3's column order for the 7
    projections of every layer is timed once after the steps."""
    import torch

    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_17733_gb300 import build as B
    from paper_2607_17733_gb300 import mxs
    if not os.path.exists(mxs.LIB_PATH):
        B.build()
    mxs.lib()
    L = args.layers or 8
    KS = [4096, 4096, 4096, 14336]
    gen = torch.Generator(device=dev)
    xs, ss = [], []
    for l in range(L):
        for ii, K in enumerate(KS):
            gen.manual_seed(SEED * 17 + rank * 10_007 + l * 11 + ii)
            x = torch.randn((CALIB_SEQ * CALIB_BATCH, K), generator=gen, device=dev, dtype=torch.float32)
            cols = torch.randperm(K, generator=gen, device=dev)[: K // 100]
            x[:, cols] *= 50.0
            xs.append(x.to(torch.bfloat16))
            ss.append(torch.zeros(K, dtype=torch.float64, device=dev))
            del x
    torch.cuda.synchronize()
    step_bytes = sum(x.numel() * 2 for x in xs)

    def fn():
        for x, sv in zip(xs, ss):
            mxs.column_sensitivity(x, s=sv, accumulate=True)

    if args.eager:
        for _ in range(args.warmup + args.steps):
            fn()
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"eager_steps": args.steps, "launches_per_step": len(xs)}), flush=True)
        return
    for _ in range(max(args.warmup, 3)):
        fn()
    torch.cuda.synchronize()
    sampler = ClockSampler(None)
    barrier(ws)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.1)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        fn()
    t1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = allreduce_max(t0.elapsed_time(t1) / args.steps, ws)
    value = ws * step_bytes / (ms * 1e-3) / 1e9
    pk = peaks()
    achieved = step_bytes / (ms * 1e-3) / 1e9  # the step is nothing but the sensitivity kernels

    # end to end: the sample's activations from pinned host memory, the sums back to the host
    hosts = [x.cpu().pin_memory() for x in xs]
    s_host = [torch.empty_like(sv, device="cpu").pin_memory() for sv in ss]
    barrier(ws)
    torch.cuda.synchronize()
    e2e_steps = max(1, min(args.steps, 10))
    t0.record()
    for _ in range(e2e_steps):
        for xh, x, sv, sh in zip(hosts, xs, ss, s_host):
            x.copy_(xh, non_blocking=True)
            mxs.column_sensitivity(x, s=sv, accumulate=True)
            sh.copy_(sv, non_blocking=True)
    t1.record()
    torch.cuda.synchronize()
    e2e_ms = allreduce_max(t0.elapsed_time(t1) / e2e_steps, ws)
    e2e = {"value": ws * step_bytes / (e2e_ms * 1e-3) / 1e9, "unit": "GB/s", "h2d_bytes_per_step": step_bytes,
           "d2h_bytes_per_step": sum(sv.numel() * 8 for sv in ss), "ms_per_step": e2e_ms}

    # Alg. 3 once: Theorem 1's R at B = 4.5 for the 7 projections of every layer
    # (layer sensitivity falling linearly from 1 to 0.3 with depth: early layers
    # are the more sensitive, Sec. 3.2), then every projection's column order
    proj_in = [0, 0, 0, 1, 2, 2, 3]  # q k v o gate up down -> input index
    d_in = [KS[i] for _ in range(L) for i in proj_in]
    s_layer = [1.0 - 0.7 * l / max(1, L - 1) for l in range(L) for _ in proj_in]
    R = mxs.allocation_r(d_in, s_layer, 4.5)
    perms = [torch.empty(K, dtype=torch.int32, device=dev) for K in d_in]
    torch.cuda.synchronize()
    t0.record()
    for l in range(L):
        for pi, ii in enumerate(proj_in):
            k = l * len(proj_in) + pi
            mxs.allocate_layer(ss[l * len(KS) + ii], R, s_layer[k], perm=perms[k])
    t1.record()
    torch.cuda.synchronize()
    alloc_ms = t0.elapsed_time(t1)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        from oracle import alloc as A
        sample = [x[:512].cpu().view(torch.int16).numpy().view(np.uint16) for x in xs[:len(KS)]]
        nbytes, t_start, passes = 0, time.perf_counter(), 0
        while True:
            for xb in sample:
                A.column_sensitivity(xb)
                nbytes += xb.size * 2
            passes += 1
            if time.perf_counter() - t_start >= 10.0:
                break
        dt = time.perf_counter() - t_start
        cpu = {"value": nbytes / dt / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"layer 0's four inputs, first 512 rows each, {passes} pass(es): numpy fp64 sum of squares",
               "seconds": dt}
    if rank == 0:
        print(json.dumps({
            "metric": "column_sensitivity_gbps", "value": value, "unit": "GB/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16 in, f32 runs + f64 sums",
            "data": "synthetic (seeded; N(0,1) with 1% of columns x50; stands in for C4 calibration samples)",
            "config": {"workload": "llama3-8b-calibration", "rows_per_step": CALIB_SEQ * CALIB_BATCH,
                       "samples_per_step": CALIB_BATCH, "layers": L,
                       "inputs_per_layer_K": KS, "l2": f"inputs larger than L2 ({step_bytes / 1e9:.2f} GB per step)"},
            "roofline": {"kernel": "column_sensitivity_kernel", "bound": "hbm", "achieved": achieved,
                         "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": achieved / pk["hbm_gbs"],
                         "peak_source": pk["source"], "traffic": None},
            "allocation": {"projections": len(d_in), "B": 4.5, "R": R, "ms": alloc_ms,
                           "kernel": "column_order_kernel (rank counting, K^2 comparisons)"},
            "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": len(xs) * args.steps, "clocks": clocks}), flush=True)


ATTN_T, ATTN_H, ATTN_HKV, ATTN_D = 4096, 32, 8, 128
ATTN_BATCHES = (1, 4, 16)


def run_attention(args):
    """Decode attention over an MXINT KV cache (the paper's KV quantization,
    4-8 bit configuration): one step = one decode token of each sequence of a
    batch, for batches of 1, 4 and 16 sequences of 4096 cached tokens, through
    the attention of `layers` LLaMA-3-8B-shaped layers (default 32; 32 query
    heads, 8 KV heads of 128 dims), one mxs_attention_decode_batch launch per
    layer and batch.  Each layer's K and V caches are quantized rows of 1024
    values with one 8-bit block (the most sensitive 32 columns) and 31 4-bit
    blocks.  Metric: GB/s of cache bytes read (codes + scales; HBM-bound), the
    step captured in a CUDA graph."""
    import torch

    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_17733_gb300 import build as B
    from paper_2607_17733_gb300 import mxs
    if not os.path.exists(mxs.LIB_PATH):
        B.build()
    mxs.lib()
    L = args.layers or 32
    T, H, Hkv, D = ATTN_T, ATTN_H, ATTN_HKV, ATTN_D
    K = Hkv * D
    gen = torch.Generator(device=dev)
    items = []  # (batch, q, kc, ks, kbits, vc, vs, vbits, out, workspace)
    for nb in ATTN_BATCHES:
        for l in range(L):
            g = I.rng(SEED, rank, 9, nb, l)
            kb = np.full(K // 32, 4, np.uint8)
            kb[g.integers(K // 32)] = 8
            vb = np.full(K // 32, 4, np.uint8)
            vb[g.integers(K // 32)] = 8
            gen.manual_seed(SEED * 19 + rank * 10_007 + nb * 101 + l)
            kx = torch.randn((nb * T, K), generator=gen, device=dev, dtype=torch.float32)
            kx[:, torch.randperm(K, generator=gen, device=dev)[: K // 100]] *= 20.0
            kc, ks, _ = mxs.quantize_act(kx.to(torch.bfloat16), kb)
            del kx
            vx = torch.randn((nb * T, K), generator=gen, device=dev, dtype=torch.float32)
            vc, vs, _ = mxs.quantize_act(vx.to(torch.bfloat16), vb)
            del vx
            q = torch.randn((nb, H, D), generator=gen, device=dev, dtype=torch.float32).to(torch.bfloat16)
            out = torch.empty((nb, H, D), dtype=torch.float32, device=dev)
            wsb = torch.zeros(mxs.attention_batch_workspace_bytes(nb, T, H, D), dtype=torch.uint8, device=dev)
            items.append((nb, q, kc, ks, kb, vc, vs, vb, out, wsb))
    torch.cuda.synchronize()
    cache_bytes = sum(t.numel() for it in items for t in (it[2], it[3], it[5], it[6]))
    step_bytes = cache_bytes + sum(it[1].numel() * 2 + it[8].numel() * 4 for it in items)
    scale = 1.0 / math.sqrt(D)

    def run(it):
        nb, q, kc, ks, kb, vc, vs, vb, out, wsb = it
        mxs.attention_decode_batch(q, Hkv, kc, ks, kb, vc, vs, vb, T, scale, out=out, workspace=wsb)

    def fn():
        for it in items:
            run(it)

    if args.eager:
        for _ in range(args.warmup + args.steps):
            fn()
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"eager_steps": args.steps, "launches_per_step": len(items)}), flush=True)
        return
    st = torch.cuda.Stream(device=dev)
    st.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(st):
        fn()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=st):
        fn()
    for _ in range(max(args.warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(None)
    barrier(ws)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.1)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        graph.replay()
    t1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = allreduce_max(t0.elapsed_time(t1) / args.steps, ws)
    value = ws * step_bytes / (ms * 1e-3) / 1e9
    pk = peaks()
    # per batch size: the same graph-free launches timed alone (device time)
    per_batch = {}
    for nb in ATTN_BATCHES:
        sub = [it for it in items if it[0] == nb]
        gb = torch.cuda.CUDAGraph()
        with torch.cuda.stream(st):
            for it in sub:
                run(it)
        torch.cuda.synchronize()
        with torch.cuda.graph(gb, stream=st):
            for it in sub:
                run(it)
        for _ in range(3):
            gb.replay()
        torch.cuda.synchronize()
        t0.record()
        for _ in range(args.steps):
            gb.replay()
        t1.record()
        torch.cuda.synchronize()
        mb = t0.elapsed_time(t1) / args.steps
        byt = sum(t.numel() for it in sub for t in (it[2], it[3], it[5], it[6]))
        per_batch[str(nb)] = {"us_per_layer": mb * 1e3 / L, "cache_gbps": byt / (mb * 1e-3) / 1e9}

    # end to end: the step's queries from pinned host memory, the outputs back
    q_host = [it[1].cpu().pin_memory() for it in items]
    o_host = [torch.empty(tuple(it[8].shape), dtype=torch.float32).pin_memory() for it in items]
    barrier(ws)
    torch.cuda.synchronize()
    e2e_steps = max(1, min(args.steps, 20))
    t0.record()
    for _ in range(e2e_steps):
        for it, qh, oh in zip(items, q_host, o_host):
            it[1].copy_(qh, non_blocking=True)
            run(it)
            oh.copy_(it[8], non_blocking=True)
    t1.record()
    torch.cuda.synchronize()
    e2e_ms = allreduce_max(t0.elapsed_time(t1) / e2e_steps, ws)
    e2e = {"value": ws * step_bytes / (e2e_ms * 1e-3) / 1e9, "unit": "GB/s",
           "h2d_bytes_per_step": sum(it[1].numel() * 2 for it in items),
           "d2h_bytes_per_step": sum(it[8].numel() * 4 for it in items), "ms_per_step": e2e_ms}

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        from oracle import attention as AT
        nb, q, kc, ks, kb, vc, vs, vb, _, _ = items[0]
        kbits = torch.randn((T, K), device=dev).to(torch.bfloat16).cpu().view(torch.int16).numpy().view(np.uint16)
        vbits = torch.randn((T, K), device=dev).to(torch.bfloat16).cpu().view(torch.int16).numpy().view(np.uint16)
        qv = q[0].float().cpu().numpy().astype(np.float64)
        kd = AT.dequantized_cache(kbits, kb)
        vd = AT.dequantized_cache(vbits, vb)
        lb = sum(t.numel() for t in (kc, ks, vc, vs)) // nb
        nbytes, t_start, passes = 0, time.perf_counter(), 0
        while True:
            AT.attention(qv, kd, vd, Hkv, scale)
            nbytes += lb
            passes += 1
            if time.perf_counter() - t_start >= 10.0:
                break
        dt = time.perf_counter() - t_start
        cpu = {"value": nbytes / dt / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"one sequence's attention in one layer over 4096 dequantized cached tokens, {passes} "
                         "pass(es) (cache dequantized once, not timed): numpy fp64", "seconds": dt}
    if rank == 0:
        print(json.dumps({
            "metric": "mxint_kv_attention_gbps", "value": value, "unit": "GB/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "MXINT codes in, bf16 MMA (exact elements), f32 sums",
            "data": "synthetic (seeded; keys N(0,1) with 1% of channels x20, values N(0,1))",
            "config": {"workload": "llama3-8b-decode-attention", "context_tokens": T, "batches": list(ATTN_BATCHES),
                       "layers": L, "heads": H, "kv_heads": Hkv, "head_dim": D,
                       "kv_map": "1 x 8-bit + 31 x 4-bit blocks",
                       "l2": f"inputs larger than L2 ({cache_bytes / 1e9:.3f} GB of cache per step)"},
            "per_batch": per_batch,
            "roofline": {"kernel": "attention_decode_kernel", "bound": "hbm",
                         "achieved": step_bytes / (ms * 1e-3) / 1e9, "peak": pk["hbm_gbs"], "unit": "GB/s",
                         "frac": step_bytes / (ms * 1e-3) / 1e9 / pk["hbm_gbs"], "peak_source": pk["source"],
                         "traffic": profile_traffic("attention.cu", "attention_decode_llama3_8b_kv4096.md")},
            "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": len(items) * args.steps, "clocks": clocks}), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.workload == "llama3-8b-prefill":
        run_prefill(args)
    elif args.workload == "llama3-8b-calibration":
        run_calibration(args)
    elif args.workload == "llama3-8b-decode-attention":
        run_attention(args)
    else:
        if args.layers is None:
            args.layers = 32
        run_ours(args)


if __name__ == "__main__":
    main()
