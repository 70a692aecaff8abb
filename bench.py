#!/usr/bin/env python
"""Benchmark of the MXINT mixed-precision linear layer (MXSens) on GB300.

Default workload (LLaMA-2-70B-shaped, the largest configuration): hidden 8192,
MLP 28672, GQA k/v 8192x1024; 80 synthetic decoder layers whose width maps
run from 60 % 4-bit (layer 0) to 95 % 4-bit (layer 79), 8-bit blocks over the
1 % outlier columns (x50) of the activations, weights N(0, 0.015).

  value (decode): for M in {1, 16} tokens, the seven projections of all 80
    layers; per decoder layer one quantizer launch + one grouped GEMM launch
    for q/k/v and for gate/up, and one fused quantize + GEMM for o and down.
    Weights are packed once (A2, 44 GB); the step is captured in a CUDA graph
    and replayed.  Metric: GB/s of algorithmic traffic (packed weights + bf16
    activations read + fp32 outputs written) per second, whole job.
  prefill (object in the same line): M = 4096 tokens through the seven
    projections of 4 layers spread over the depth (0, 26, 53, 79); per stage
    of projections that read one hidden state one quantizer launch to MMA
    planes, then the tcgen05 GEMMs.  Effective TOPS = 2*M*N*K per second,
    with the GEMMs' roofline and the quantizer's HBM roofline.

--workload also offers the LLaMA-3-8B decode / prefill / calibration / KV
attention workloads.  --impl reference times the CPU oracle (the paper
publishes no kernel to run) on a bounded sample of the same workload, on the
host cores.
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

SEED = 2607
STAGES = [[0, 1, 2], [3], [4, 5], [6]]  # q k v | o | gate up | down: the projections of a stage share an input


class Spec:
    """A decode or prefill workload: the model's projection shapes, how many
    decoder layers, the width map of each projection, the weight and
    activation distributions."""

    def __init__(self, name, shapes, layers, Ms, w_sigma, outlier_frac, outlier_scale, map_fn, student_t=False,
                 layer_ids=None, sample_cols=2048):
        self.name, self.shapes, self.layers, self.Ms = name, shapes, layers, tuple(Ms)
        self.w_sigma, self.outlier_frac, self.outlier_scale = w_sigma, outlier_frac, outlier_scale
        self.map_fn, self.student_t = map_fn, student_t
        self.layer_ids = list(layer_ids) if layer_ids is not None else list(range(layers))
        self.sample_cols = sample_cols

    def bits(self, rank, l, pi, K):
        return self.map_fn(K, l, self.layers, I.rng(SEED, rank, 70, l, pi))


def _map_8b_decode(K, l, L, g):
    return I.width_map(K // 32, 0.85, 0.10, 0.05, g)


def _map_8b_prefill(K, l, L, g):
    return I.width_map(K // 32, 0.80, 0.15, 0.05, g)


def _map_70b(K, l, L, g):
    return I.llama70b_layer_map(K, l, L, g)


def spec_for(workload: str, layers=None) -> Spec:
    if workload == "llama3-8b-decode":
        return Spec("llama3-8b-decode", I.LLAMA3_8B, layers or 32, (1, 4, 16), 0.02, 0.01, 30.0, _map_8b_decode)
    if workload == "llama3-8b-prefill":
        return Spec("llama3-8b-prefill", I.LLAMA3_8B, layers or 8, (2048,), 0.02, 0.005, None, _map_8b_prefill,
                    student_t=True, sample_cols=1024)
    if workload == "llama2-70b-decode":
        return Spec("llama2-70b-decode", I.LLAMA2_70B, layers or 80, (1, 16), 0.015, 0.01, 50.0, _map_70b,
                    sample_cols=512)
    if workload == "llama2-70b-prefill":
        L = layers or 80
        ids = sorted({int(round(v)) for v in np.linspace(0, L - 1, min(4, L))})
        return Spec("llama2-70b-prefill", I.LLAMA2_70B, L, (4096,), 0.015, 0.01, 50.0, _map_70b,
                    layer_ids=ids, sample_cols=512)
    raise ValueError(workload)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--layers", type=int, default=None,
                    help="decoder layers of the model (default 80 for LLaMA-2-70B, 32 for LLaMA-3-8B decode, "
                         "8 for LLaMA-3-8B prefill)")
    ap.add_argument("--workload", default="llama2-70b",
                    choices=["llama2-70b", "llama3-8b-decode", "llama3-8b-prefill", "llama3-8b-calibration",
                             "llama3-8b-decode-attention"])
    ap.add_argument("--part", default="both", choices=["both", "decode", "prefill"],
                    help="llama2-70b: run the decode part, the prefill part or both (one JSON line)")
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


def code_sha(src: bytes) -> str:
    """sha256[:16] of a CUDA source with its comments and blank space removed:
    the same for two versions that differ only in comments or layout."""
    import hashlib
    import re
    text = src.decode("utf-8")
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return hashlib.sha256(" ".join(text.split()).encode()).hexdigest()[:16]


def profile_traffic(kernel_file: str, profile_md: str):
    """DRAM bytes per launch recorded in a committed ncu summary, if it was taken
    on the current code of the kernel: the summary's sha is the sha256[:16] of
    the .cu file, or of its code alone (code_sha)."""
    import hashlib
    try:
        src = open(os.path.join(ROOT, "paper_2607_17733_gb300", "csrc", kernel_file), "rb").read()
        text = open(os.path.join(ROOT, "profiles", profile_md)).read()
    except OSError:
        return None
    shas = {hashlib.sha256(src).hexdigest()[:16], code_sha(src)}
    for line in text.splitlines():
        if line.startswith("traffic_bytes_per_launch:"):
            parts = line.split()
            # traffic_bytes_per_launch: <bytes> kernel_sha: <sha>
            if len(parts) >= 4 and parts[3] in shas:
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
_SAMPLES = {}


def _oracle_jobs(spec: Spec, seed_rank: int = 0):
    """The first timed layer of `spec` for the oracle: every projection's
    first min(N, spec.sample_cols) output columns, weights quantized once
    (offline packing is not timed), activations for every M of the spec (the
    first 64 token rows of a prefill M)."""
    key = (spec.name, seed_rank)
    if key not in _SAMPLES:
        from oracle import mxo
        jobs = []
        l = spec.layer_ids[0]
        for pi, (name, K, N) in enumerate(spec.shapes):
            bits = spec.bits(seed_rank, l, pi, K)
            N = min(N, spec.sample_cols)
            w = I.normal_bf16((N, K), spec.w_sigma, I.rng(SEED, seed_rank, 71, l, pi))
            w_s, w_c = mxo.quantize_bf16(w, bits)
            del w
            for M in spec.Ms:
                Ms = min(M, 64)
                x = I.activations_bf16(Ms, bits, I.rng(SEED, seed_rank, 72, pi, M), spec.outlier_frac,
                                       outlier_scale=spec.outlier_scale, student_t=spec.student_t)
                jobs.append((bits, x, w_s, w_c, K, N, Ms))
        _SAMPLES[key] = jobs
    return _SAMPLES[key]


def oracle_sample(spec: Spec, min_seconds: float = 10.0):
    """Time the oracle on a bounded sample of the step: the activation
    quantization and exact GEMM of the jobs of _oracle_jobs, passes repeated
    until min_seconds have elapsed (at least one).  Returns (rate, seconds,
    threads, text, unit): GB/s of the same algorithmic traffic as the GPU
    step for decode, effective TOPS for prefill."""
    from oracle import mxo
    jobs = _oracle_jobs(spec)
    t0 = time.perf_counter()
    nbytes = ops = passes = 0
    while True:
        for bits, x, w_s, w_c, K, N, M in jobs:
            a_s, a_c = mxo.quantize_bf16(x, bits)
            mxo.gemm(bits, a_c, a_s, w_c, w_s)
            n4 = int(np.sum(bits == 4))
            nbytes += N * (16 * n4 + 32 * (bits.size - n4) + bits.size) + M * K * 2 + M * N * 4
            ops += 2 * M * N * K
        passes += 1
        if time.perf_counter() - t0 >= min_seconds:
            break
    dt = time.perf_counter() - t0
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    decode = spec.Ms[0] <= 16
    desc = (f"layer {spec.layer_ids[0]} of {spec.name} (q/k/v/o/gate/up/down, first min(N,{spec.sample_cols}) "
            "output columns" + (f") at M={','.join(map(str, spec.Ms))}" if decode else
                                f", first 64 of {spec.Ms[0]} token rows)") +
            f", {passes} pass(es): oracle activation quantization + exact GEMM, OpenMP over output rows")
    if decode:
        return nbytes / dt / 1e9, dt, threads, desc, "GB/s"
    return ops / dt / 1e12, dt, threads, desc, "TOPS"


def reference_spec(args) -> Spec | None:
    if args.workload == "llama2-70b":
        return spec_for("llama2-70b-prefill" if args.part == "prefill" else "llama2-70b-decode", args.layers)
    if args.workload in ("llama3-8b-decode", "llama3-8b-prefill"):
        return spec_for(args.workload, args.layers)
    return None


def run_reference(args):
    ws, rank, _ = dist_setup()
    if rank != 0:
        return
    spec = reference_spec(args)
    if spec is None:
        print(json.dumps({"impl": "reference", "unavailable": f"the oracle arm times the GEMM workloads "
                          f"(llama2-70b, llama3-8b-decode, llama3-8b-prefill), not {args.workload}"}), flush=True)
        return
    for _ in range(args.warmup):
        oracle_sample(spec, min_seconds=0.0)
    vals, secs = [], []
    desc, threads, unit = "", 1, "GB/s"
    for _ in range(args.steps):
        v, dt, threads, desc, unit = oracle_sample(spec, min_seconds=0.0)
        vals.append(v)
        secs.append(dt)
    value = statistics.median(vals)
    decode = unit == "GB/s"
    line = {
        "impl": "reference", "metric": "mxint_decode_gemm_gbps" if decode else "mxint_prefill_gemm_tops",
        "value": value, "unit": unit,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * statistics.median(secs), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int64+f64", "data": "synthetic",
        "config": {"workload": args.workload, "M": list(spec.Ms), "layers": spec.layers,
                   "sample": desc},
        "cpu_baseline": {"value": value, "unit": unit, "cores": threads, "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------- GPU arm
def _gpu_setup():
    import torch
    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_17733_gb300 import build as B
    from paper_2607_17733_gb300 import mxs
    if not os.path.exists(mxs.LIB_PATH):
        B.build()
    mxs.lib()
    return torch, ws, rank, dev


def _weight(torch, gen, dev, N, K, sigma, seed):
    gen.manual_seed(seed)
    return (torch.randn((N, K), generator=gen, device=dev, dtype=torch.float32) * sigma).to(torch.bfloat16)


def run_decode(args, spec: Spec):
    """Decode step of `spec`: for every M of the spec, the seven projections of
    every layer (A1 + A4), weights packed once (A2), the step captured in a
    CUDA graph.  Returns the JSON line (rank 0) or None."""
    torch, ws, rank, dev = _gpu_setup()
    from paper_2607_17733_gb300 import mxs
    from paper_2607_17733_gb300.runtime import MxLinear

    L = spec.layers
    # ---- weights: drawn on the GPU (seeded per layer/projection), packed once
    layers = []
    gen = torch.Generator(device=dev)
    for l in range(L):
        projs = []
        for pi, (name, K, N) in enumerate(spec.shapes):
            w = _weight(torch, gen, dev, N, K, spec.w_sigma, SEED * 1_000_003 + rank * 10_007 + l * 101 + pi)
            projs.append(MxLinear(w, spec.bits(rank, l, pi, K)))
            del w
        layers.append(projs)
    torch.cuda.synchronize()

    # ---- inputs: one contiguous pinned host block and one device block per step
    items = []  # (M, lin, x_dev, bufs)
    x_total = sum(M * lin.K for M in spec.Ms for projs in layers for lin in projs)
    x_host = torch.empty(x_total, dtype=torch.bfloat16, pin_memory=True)
    x_dev = torch.empty_like(x_host, device=dev)
    y_sizes = []
    off = 0
    for M in spec.Ms:
        for l in range(L):
            for pi, lin in enumerate(layers[l]):
                xb = I.activations_bf16(M, lin.bits, I.rng(SEED, rank, 2, M, l, pi), spec.outlier_frac,
                                        outlier_scale=spec.outlier_scale)
                n = M * lin.K
                x_host[off:off + n].copy_(torch.from_numpy(xb.view(np.int16).ravel()).view(torch.bfloat16))
                items.append((M, lin, x_dev[off:off + n].view(M, lin.K), lin.buffers(M, dev)))
                y_sizes.append(M * lin.N)
                off += n
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
    nproj = len(spec.shapes)
    # M = 1 through mxs_linear_decode(_group): one kernel (quantization fused);
    # otherwise a quantizer launch and a GEMM launch
    per_gemm = {M: (1 if (M == 1 and args.path in ("fused", "grouped")) else 2) for M in spec.Ms}
    launches_per_step = sum(per_gemm[M] for M, _, _, _ in items)
    gemm_launches = len(items)
    if args.path == "grouped":  # per stage one GEMM launch, after one quantizer launch when M > 1
        launches_per_step = sum(per_gemm[M] for M in spec.Ms) * spec.layers * len(STAGES)
        gemm_launches = len(items) // nproj * len(STAGES)

    # ---- the step as one CUDA graph.  Inputs are independent synthetic draws, so
    # for each M the graph runs all activation quantizations, then all GEMMs;
    # on one stream every kernel waits for the previous one either way.  Two
    # event nodes per M bracket the GEMM segment: the dominant kernel's time
    # is read from them for every timed step.
    capture_stream = torch.cuda.Stream(device=dev)
    groups = [[it for it in items if it[0] == M] for M in spec.Ms]

    def make_step(events=None, grps=None):
        grps = groups if grps is None else grps

        def fn():
            for gi, grp in enumerate(grps):
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
                    for base in range(0, len(grp), nproj):
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
        return None

    plain = capture(make_step())
    try:
        ev_sets = [[(torch.cuda.Event(enable_timing=True, external=True),
                     torch.cuda.Event(enable_timing=True, external=True)) for _ in groups]
                   for _ in range(args.steps)]
        timed = [capture(make_step(evs)) for evs in ev_sets]
    except TypeError:  # torch without external events: time the plain graph only
        ev_sets, timed = None, [plain] * args.steps

    for _ in range(max(args.warmup, 3)):
        plain.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(_gpu_uuid(torch, dev))

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
    ms = allreduce_max(t0.elapsed_time(t1) / args.steps, ws)
    value = ws * step_bytes / (ms * 1e-3) / 1e9
    tops = ws * step_ops / (ms * 1e-3) / 1e12

    # ---- the dominant kernel (decode GEMM): per-launch durations from the graphs' events
    pk = peaks()
    roofline = None
    if ev_sets is not None:
        gemm_ms = sum(s.elapsed_time(e) for evs in ev_sets for s, e in evs) / len(ev_sets)  # per step
        achieved = gemm_bytes / (gemm_ms * 1e-3) / 1e9
        prof = "gemm_decode_llama2_70b_decode.md" if spec.name.startswith("llama2-70b") \
            else "gemm_decode_llama3_8b_decode.md"
        fused = args.path in ("fused", "grouped")
        roofline = {"kernel": ("gemv_decode_kernel for M = 1 (quantization fused), decode_tc_kernel after "
                               "quantize_act_kernel (PDL chain) for M > 1" if fused
                               else f"gemm_decode_kernel ({args.path} path)"),
                    "bound": "hbm", "achieved": achieved,
                    "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": achieved / pk["hbm_gbs"],
                    "peak_source": pk["source"] + " (HBM copy)",
                    "traffic": profile_traffic("decode_tc.cu" if fused else "gemm_decode.cu", prof),
                    "bytes_per_step": gemm_bytes, "gemm_ms_per_step": gemm_ms,
                    "gemm_launches_per_step": gemm_launches, "share_of_step": gemm_ms / ms}

    # ---- end to end through the public API with host buffers: every step copies
    # its inputs in from pinned host memory and reads its outputs back, on two
    # copy streams (in, out) beside the compute stream, over two device buffer
    # sets, so that step k+1's inputs arrive and step k's outputs leave while
    # the neighbouring step computes (the copies share the host link and HBM)
    x_dev2, y_dev2 = torch.empty_like(x_dev), torch.empty_like(y_dev)

    def rebind(it):
        M, lin, x, bufs = it
        xo = (x.data_ptr() - x_dev.data_ptr()) // x.element_size()
        yo = (bufs["y"].data_ptr() - y_dev.data_ptr()) // 4
        b2 = dict(bufs)
        b2["y"] = y_dev2[yo:yo + M * lin.N].view(M, lin.N)
        return (M, lin, x_dev2[xo:xo + M * lin.K].view(M, lin.K), b2)

    plain2 = capture(make_step(grps=[[rebind(it) for it in grp] for grp in groups]))
    sets = [(x_dev, y_dev, plain), (x_dev2, y_dev2, plain2)]
    comp, s_in, s_out = torch.cuda.current_stream(), torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    got = [torch.cuda.Event() for _ in sets]   # a set's inputs are in
    done = [torch.cuda.Event() for _ in sets]  # a set's compute is done
    out = [torch.cuda.Event() for _ in sets]   # a set's outputs are out
    barrier(ws)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e2e_steps = max(1, min(args.steps, 50))
    e0.record(comp)
    s_in.wait_event(e0)
    s_out.wait_event(e0)
    for k in range(e2e_steps):
        b = k % 2
        xd, yd, g = sets[b]
        if k >= 2:
            s_in.wait_event(done[b])  # step k - 2 has read this set's inputs
        with torch.cuda.stream(s_in):
            xd.copy_(x_host, non_blocking=True)
        got[b].record(s_in)
        comp.wait_event(got[b])
        if k >= 2:
            comp.wait_event(out[b])  # step k - 2's outputs have left this set
        g.replay()
        done[b].record(comp)
        s_out.wait_event(done[b])
        with torch.cuda.stream(s_out):
            y_host.copy_(yd, non_blocking=True)
        out[b].record(s_out)
    comp.wait_stream(s_in)
    comp.wait_stream(s_out)
    e1.record(comp)
    torch.cuda.synchronize()
    e2e_ms = allreduce_max(e0.elapsed_time(e1) / e2e_steps, ws)
    e2e = {"value": ws * step_bytes / (e2e_ms * 1e-3) / 1e9, "unit": "GB/s",
           "h2d_bytes_per_step": x_host.numel() * 2, "d2h_bytes_per_step": y_host.numel() * 4,
           "ms_per_step": e2e_ms}

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, dt, threads, desc, unit = oracle_sample(spec)
        cpu = {"value": v, "unit": unit, "cores": threads, "kind": "oracle", "sample": desc, "seconds": dt}
    w_bytes = sum(lin.weight_bytes for p in layers for lin in p)
    del plain, timed, layers, items, x_dev, y_dev
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if rank != 0:
        return None
    maps = ("4-bit share from 60% (layer 0) to 95% (last layer), 8-bit blocks over the 1% outlier columns, "
            "the rest 6-bit" if spec.map_fn is _map_70b else "85/10/5 % (4/6/8 bits)")
    return {
        "metric": "mxint_decode_gemm_gbps", "value": value, "unit": "GB/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8+f32",
        "data": f"synthetic (seeded; weights N(0,{spec.w_sigma}), activations N(0,1) with "
                f"{100 * spec.outlier_frac:g}% outlier columns x{spec.outlier_scale:g})",
        "config": {"workload": spec.name, "M": list(spec.Ms), "layers": L,
                   "path": {"planes": "quantize to MMA planes, then GEMM over the planes (TMA)",
                            "fused": "mxs_linear_decode: quantize + GEMM chained by programmatic dependent launch",
                            "grouped": "mxs_linear_decode_group for q/k/v and gate/up (one GEMM launch per "
                                       "group), mxs_linear_decode for o, down; M = 1: the CUDA-core GEMM with "
                                       "the quantization fused, else one quantizer launch before each tensor-core GEMM",
                            "codes": "quantize to packed codes, GEMM over the codes"}[args.path],
                   "projections": [p[0] for p in spec.shapes], "maps": maps,
                   "parallelism": f"replicas x{ws}", "l2": "inputs larger than L2 (packed weights "
                   f"{w_bytes / 1e9:.2f} GB per M per step)"},
        "tops": tops,
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
    }


def _gpu_uuid(torch, dev):
    try:
        return "GPU-" + str(torch.cuda.get_device_properties(dev).uuid).replace("GPU-", "")
    except Exception:
        return None


def probe_peaks(torch):
    """Tensor-core rates measured on this GPU with mxs_probe_mma (one CTA per
    SM, back-to-back MMAs over zero operands, best of three launches): the
    block-scaled FP8 MMA the prefill GEMM issues for 4-bit blocks, the bf16
    MMA it issues for 6/8-bit blocks (both M = 128, N = 256), and the legacy
    mma.sync s8 rate (this part's INT8 tensor path).  TFLOP/s (TOPS for s8)."""
    from paper_2607_17733_gb300 import mxs
    out = {}
    for name, kind, n, iters in (("fp8_block_scaled_tflops", mxs.PROBE_FP8, 256, 20000),
                                 ("bf16_tflops", mxs.PROBE_BF16, 256, 20000),
                                 ("s8_mma_sync_tops", mxs.PROBE_S8_MMA_SYNC, 16, 100000)):
        for _ in range(2):
            mxs.probe_mma(kind, n, iters)
        torch.cuda.synchronize()
        best = 0.0
        for _ in range(3):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            flop = mxs.probe_mma(kind, n, iters)
            e1.record()
            torch.cuda.synchronize()
            best = max(best, flop / (e0.elapsed_time(e1) * 1e-3) / 1e12)
        out[name] = best
    if mxs.probe_status(reset=True) != 0:
        return {}
    return out


def run_prefill_part(args, spec: Spec):
    """Prefill step of `spec` (M = spec.Ms[0] tokens) through the seven
    projections of the layers spec.layer_ids.  Per stage of a layer (q/k/v,
    o, gate/up, down: the projections of a stage read one hidden state): one
    quantizer launch to MMA planes (A1) for its projections, then their
    tcgen05 GEMMs (A3).  Metric: effective TOPS = 2*M*N*K / s, whole job.
    Returns the JSON object (rank 0) or None."""
    torch, ws, rank, dev = _gpu_setup()
    from paper_2607_17733_gb300 import mxs
    from paper_2607_17733_gb300.runtime import MxLinear
    M = spec.Ms[0]
    gen = torch.Generator(device=dev)
    items = []
    for l in spec.layer_ids:
        for pi, (name, K, N) in enumerate(spec.shapes):
            w = _weight(torch, gen, dev, N, K, spec.w_sigma, SEED * 7 + rank * 10_007 + l * 101 + pi)
            bits = spec.bits(rank, l, pi, K)
            items.append((MxLinear(w, bits, with_planes=True), bits))
            del w
    xs, planes, ys = [], [], []
    for idx, (lin, bits) in enumerate(items):
        # N(0,1) activations with outlier columns inside the 8-bit blocks: scaled,
        # or redrawn from a Student-t(3) = Z / sqrt(chi2_3 / 3); drawn on the GPU
        gen.manual_seed(SEED * 13 + rank * 10_007 + idx)
        x = torch.randn((M, lin.K), generator=gen, device=dev, dtype=torch.float32)
        n_out = int(np.floor(spec.outlier_frac * lin.K + 0.5))
        cols = torch.from_numpy(I.outlier_columns(bits, n_out, I.rng(SEED, rank, 6, idx))).to(dev)
        if spec.student_t:
            z = torch.randn((M, cols.numel(), 4), generator=gen, device=dev, dtype=torch.float32)
            x[:, cols] = z[..., 0] / torch.sqrt((z[..., 1:] ** 2).sum(-1) / 3.0)
        else:
            x[:, cols] *= spec.outlier_scale
        xs.append(x.to(torch.bfloat16))
        del x
        planes.append(torch.empty(mxs.act_planes_bytes(M, lin.K, bits), dtype=torch.uint8, device=dev))
        ys.append(torch.empty((M, lin.N), dtype=torch.float32, device=dev))
    torch.cuda.synchronize()
    nproj = len(spec.shapes)
    step_ops = sum(2 * M * lin.N * lin.K for lin, _ in items)
    # tensor work as issued: a 4-bit K' stage is four K=32 FP8 MMAs, a 6/8-bit stage
    # four K=16 bf16 MMAs of the same cost: 2*M*N*128 per K' stage, in FP8 units
    nst = []
    for lin, bits in items:
        n4 = int(np.sum(bits == 4))
        nst.append((n4 + 3) // 4 + (bits.size - n4 + 1) // 2)
    issued_ops = sum(2 * M * lin.N * 128 * s for (lin, _), s in zip(items, nst))
    q_bytes = sum(2 * M * lin.K + pl.numel() for (lin, _), pl in zip(items, planes))
    n_launch = len(items) + len(items) // nproj * len(STAGES)

    def fn(events=None, xs=xs, ys=ys):
        for base in range(0, len(items), nproj):
            for si, stage in enumerate(STAGES):
                idxs = [base + i for i in stage]
                if events is not None:
                    events["q"][base // nproj * len(STAGES) + si][0].record()
                if len(idxs) == 1:
                    mxs.quantize_act(xs[idxs[0]], items[idxs[0]][1], planes=planes[idxs[0]], want_codes=False)
                else:
                    mxs.quantize_act_group([(xs[i], items[i][1], planes[i]) for i in idxs])
                if events is not None:
                    events["q"][base // nproj * len(STAGES) + si][1].record()
                for idx in idxs:
                    lin, bits = items[idx]
                    if events is not None:
                        events["g"][idx][0].record()
                    mxs.gemm_prefill(planes[idx], bits, lin.packed, M, lin.N, y=ys[idx])
                    if events is not None:
                        events["g"][idx][1].record()

    if args.eager:
        for _ in range(args.warmup + args.steps):
            fn()
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"eager_steps": args.steps, "launches_per_step": n_launch}), flush=True)
        return None
    for _ in range(max(args.warmup, 3)):
        fn()
    torch.cuda.synchronize()

    def evpair():
        return (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))

    steps = max(1, min(args.steps, 20))
    evs = [{"g": [evpair() for _ in items], "q": [evpair() for _ in range(len(items) // nproj * len(STAGES))]}
           for _ in range(steps)]
    sampler = ClockSampler(_gpu_uuid(torch, dev))
    barrier(ws)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.1)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for k in range(steps):
        fn(evs[k])
    t1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = allreduce_max(t0.elapsed_time(t1) / steps, ws)
    gemm_ms = sum(s.elapsed_time(e) for ev in evs for s, e in ev["g"]) / steps
    quant_ms = sum(s.elapsed_time(e) for ev in evs for s, e in ev["q"]) / steps
    pk = peaks()
    fp8_peak = 2.0 * pk["bf16_tflops"]
    achieved = step_ops / (gemm_ms * 1e-3) / 1e12
    issued = issued_ops / (gemm_ms * 1e-3) / 1e12
    value = ws * step_ops / (ms * 1e-3) / 1e12
    q_gbs = q_bytes / (quant_ms * 1e-3) / 1e9

    probes = probe_peaks(torch) if rank == 0 else {}

    # end to end: every step's activations from pinned host memory and every
    # output back, on an input and an output copy stream beside the compute
    # stream over two device buffer sets (as in the decode part)
    x_host = [x.cpu().pin_memory() for x in xs]
    y_host = [torch.empty(tuple(y.shape), dtype=torch.float32).pin_memory() for y in ys]
    sets = [(xs, ys), ([torch.empty_like(x) for x in xs], [torch.empty_like(y) for y in ys])]
    comp, s_in, s_out = torch.cuda.current_stream(), torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    got = [torch.cuda.Event() for _ in sets]   # a set's inputs are in
    done = [torch.cuda.Event() for _ in sets]  # a set's compute is done
    out = [torch.cuda.Event() for _ in sets]   # a set's outputs are out
    barrier(ws)
    torch.cuda.synchronize()
    e2e_steps = max(1, min(steps, 5))
    t0.record(comp)
    s_in.wait_event(t0)
    s_out.wait_event(t0)
    for k in range(e2e_steps):
        b = k % 2
        X, Y = sets[b]
        if k >= 2:
            s_in.wait_event(done[b])  # step k - 2 has read this set's inputs
        with torch.cuda.stream(s_in):
            for xh, x in zip(x_host, X):
                x.copy_(xh, non_blocking=True)
        got[b].record(s_in)
        comp.wait_event(got[b])
        if k >= 2:
            comp.wait_event(out[b])  # step k - 2's outputs have left this set
        fn(xs=X, ys=Y)
        done[b].record(comp)
        s_out.wait_event(done[b])
        with torch.cuda.stream(s_out):
            for yh, y in zip(y_host, Y):
                yh.copy_(y, non_blocking=True)
        out[b].record(s_out)
    comp.wait_stream(s_in)
    comp.wait_stream(s_out)
    t1.record(comp)
    torch.cuda.synchronize()
    e2e_ms = allreduce_max(t0.elapsed_time(t1) / e2e_steps, ws)
    e2e = {"value": ws * step_ops / (e2e_ms * 1e-3) / 1e12, "unit": "TOPS",
           "h2d_bytes_per_step": sum(x.numel() * 2 for x in xs), "d2h_bytes_per_step": sum(y.numel() * 4 for y in ys),
           "ms_per_step": e2e_ms}
    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, dt, threads, desc, unit = oracle_sample(spec)
        cpu = {"value": v, "unit": unit, "cores": threads, "kind": "oracle", "sample": desc, "seconds": dt}
    q_launches = len(items) // nproj * len(STAGES)
    del items, xs, planes, ys, x_host, y_host, sets
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if rank != 0:
        return None
    prof = "gemm_prefill_llama2_70b_prefill.md" if spec.name.startswith("llama2-70b") \
        else "gemm_prefill_llama3_8b_prefill.md"
    return {
        "metric": "mxint_prefill_gemm_tops", "value": value, "unit": "TOPS", "n_gpus": ws,
        "steps": steps, "warmup": max(args.warmup, 3), "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "e4m3 (4-bit blocks) + bf16 (6/8-bit blocks), f32 accumulation",
        "data": f"synthetic (seeded; W N(0,{spec.w_sigma}), A N(0,1) with " +
                ("Student-t(3) outlier channels" if spec.student_t else f"outlier columns x{spec.outlier_scale:g}") +
                f" on {100 * spec.outlier_frac:g}% of K)",
        "config": {"workload": spec.name, "M": M, "layers": spec.layer_ids, "of_layers": spec.layers,
                   "l2": "inputs larger than L2"},
        "roofline": {"kernel": "gemm_prefill_kernel", "bound": "tensor", "achieved": achieved,
                     "peak": fp8_peak, "unit": "TFLOP/s", "frac": achieved / fp8_peak,
                     "peak_source": pk["source"] + " bf16 x 2 (fp8/bf16 nominal ratio)",
                     "issued_fp8_equivalent": issued, "issued_frac": issued / fp8_peak,
                     "probe": probes,
                     "frac_of_probe_fp8": achieved / probes["fp8_block_scaled_tflops"] if probes else None,
                     "issued_frac_of_probe_fp8": issued / probes["fp8_block_scaled_tflops"] if probes else None,
                     "frac_of_s8_mma_sync": achieved / probes["s8_mma_sync_tops"] if probes else None,
                     "traffic": profile_traffic("gemm_prefill.cu", prof),
                     "gemm_ms_per_step": gemm_ms, "share_of_step": gemm_ms / ms},
        "quantizer": {"kernel": "quantize_act_group_kernel / quantize_act_kernel (bf16 in, MMA planes out)",
                      "bound": "hbm", "achieved": q_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                      "frac": q_gbs / pk["hbm_gbs"], "bytes_per_step": q_bytes, "ms_per_step": quant_ms,
                      "launches_per_step": q_launches},
        "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": n_launch * steps, "clocks": clocks}


def run_llama70b(args):
    """The default workload: LLaMA-2-70B decode (the line's value) and
    prefill (its `prefill` object)."""
    line = None
    if args.part in ("both", "decode"):
        line = run_decode(args, spec_for("llama2-70b-decode", args.layers))
    if args.part in ("both", "prefill"):
        pre = run_prefill_part(args, spec_for("llama2-70b-prefill", args.layers))
        if line is None:
            line = pre
        elif pre is not None:
            line["prefill"] = pre
    if line is not None:
        if "config" in line:
            line["config"]["workload"] = "llama2-70b" + ("" if args.part == "both" else f" ({args.part})")
        print(json.dumps(line), flush=True)


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
    elif args.workload == "llama2-70b":
        run_llama70b(args)
    elif args.workload == "llama3-8b-prefill":
        line = run_prefill_part(args, spec_for("llama3-8b-prefill", args.layers))
        if line is not None:
            print(json.dumps(line), flush=True)
    elif args.workload == "llama3-8b-calibration":
        run_calibration(args)
    elif args.workload == "llama3-8b-decode-attention":
        run_attention(args)
    else:
        line = run_decode(args, spec_for("llama3-8b-decode", args.layers))
        if line is not None:
            print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
