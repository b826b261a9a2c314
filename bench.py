#!/usr/bin/env python3
"""Benchmark of the SPHQuant decode GEMV on GB300 (one JSON line on stdout).

Workload (one "step" = one pass of the hot path over one batch of input):
  1. the batch-1 W2/W3 GEMV sweep at 4096x4096 and 8192x8192.  Each shape has
     a pool of distinct packed matrices whose total size exceeds twice the L2
     cache, and a step runs one GEMV on every matrix of every pool, so every
     GEMV streams its codes from HBM;
  2. one token through the 28-layer x 7-projection linear stack of a
     7B-class decoder at W2 and at W3 (196 distinct matrices each, batch 1).
  Each pool and each stack is captured once as a CUDA graph of back-to-back
  launches on one stream.  The sweep's matrices carry encoder codes: the
  library's GPU encoder (sphq_encode) run on seeded Gaussian weights with
  outliers (the encoded configuration); the stacks carry seeded uniformly
  random codes, as the decoder configurations specify.

value    = algorithmic bytes of all GEMVs of a step / device time per step (GB/s)
sweep    = per shape: us per GEMV, GB/s and fraction of HBM (CUDA events
           around each pool's graph)
stack    = us per token for the W2 and W3 stacks (CUDA events around each)
stack_fused = the same stacks with q|k|v and gate|up fused by row
           concatenation (4 GEMVs per layer), timed after the steps
roofline = the dominant kernel's algorithmic bytes per launch / its average
           launch time (CUDA events on the launching stream), against the
           measured HBM copy bandwidth
e2e      = the same metric through sphq_gemv_host (pinned host x in, y out,
           copies inside the timed region), one GEMV per sweep shape per step
clocks   = nvidia-smi samples taken while the timed steps run

--impl reference runs the float64 CPU oracle (the reference arm of this
build) on bounded row samples of the same workload.
"""
from __future__ import annotations

import argparse
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

import sphq_inputs as inp  # noqa: E402

METRIC = "batch-1 W2/W3 GEMV effective GB/s and % of GB300 HBM peak; µs/token for linear stack"
WORKLOAD = ("W2+W3 GEMV sweep 4096^2 and 8192^2 + 28-layer W2/W3 decoder linear stack, "
            "batch 1")
UNIT = "GB/s"

# DRAM traffic of the GEMV kernel per launch relative to its algorithmic bytes,
# from one-pass ncu captures (dram__bytes_read.sum + dram__bytes_write.sum) of
# the 8192x8192 batch-1 launches, valid for the kernel sources with this
# digest only; the roofline reports traffic null otherwise.
TRAFFIC_SOURCES = ("paper_2609_24875_gb300/csrc/sphq_gemv_kernel.cuh",
                   "paper_2609_24875_gb300/csrc/sphq_gemv.cu",
                   "paper_2609_24875_gb300/csrc/sphq_layout.cuh")
TRAFFIC_DIGEST = "0db785fb6516774e:aee7ee8072d8a4f1:4e816d7cd02affb6"
TRAFFIC_RATIO = {2: 21040640 / 21005312, 3: 28536064 / 28475392}


def kernel_digest() -> str:
    import hashlib
    out = []
    for rel in TRAFFIC_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            out.append(hashlib.sha256(f.read()).hexdigest()[:16])
    return ":".join(out)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []  # (host time, csv line)
        self.window = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "10"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (FileNotFoundError, OSError):
            self.proc = None
        time.sleep(1.0)  # nvidia-smi start-up; samples before the window are dropped
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.perf_counter(), line.strip()))

    def mark(self, t0: float, t1: float):
        """Host times bracketing the timed region (enqueue .. synchronize)."""
        self.window = (t0, t1)

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.t.join(timeout=2)

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ts, ln in self.lines:
            if self.window is not None and not (self.window[0] <= ts <= self.window[1]):
                continue
            p = [t.strip() for t in ln.split(",")]
            if len(p) < 8:
                continue
            try:
                sm.append(float(p[0]))
                mx.append(float(p[1]))
            except ValueError:
                continue
            for n, v in zip(names, p[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# distributed (replicas only: every rank runs its own pools)
# ---------------------------------------------------------------------------

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def dist_barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def dist_max(world, v: float) -> float:
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def l2_bytes() -> int:
    import torch
    p = torch.cuda.get_device_properties(torch.cuda.current_device())
    return int(getattr(p, "L2_cache_size", 0) or getattr(p, "l2_cache_size", 0) or 128 << 20)


def make_pool(bits: int, rows: int, cols: int, n: int, seed: int, dev):
    """n distinct device copies of one seeded matrix (distinct buffers, so no
    L2 reuse between consecutive GEMVs)."""
    import torch

    from paper_2609_24875_gb300 import SphqMatrix
    codes, x = inp.random_codes(bits, rows, cols, seed=seed)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)
    cb, sc, of = t(codes.codebook), t(codes.scale), t(codes.offset)
    sg, ix, rc = t(codes.sign), t(codes.idx), t(codes.rcode)
    mats = []
    for _ in range(n):
        m = SphqMatrix(rows, cols, bits, cb, sc, of)
        m.pack(sg, ix, rc)
        mats.append(m)
    del sg, ix, rc
    xd = t(x).view(torch.float16)
    return mats, xd, codes, x


def make_encoded_pool(bits: int, n: int, P: int, seed: int, dev):
    """P distinct device copies of one n x n matrix whose codes come from the
    library's GPU encoder (sphq_encode, Eqs. (3), (5)-(7)) run on seeded
    Gaussian weights N(0, 0.02^2) with 0.1% of the scalars x20 -- the encoded
    configuration's recipe (sphq_inputs.gaussian_weights), with the random
    positive-unit codebook and N(0, 1) activations of sphq_inputs.
    Returns (mats, x on the device, host x)."""
    import torch

    from paper_2609_24875_gb300 import SphqMatrix
    cb, x = inp.encoded_inputs_rng(bits, n, seed=seed)
    w = torch.from_numpy(inp.gaussian_weights(n, n, seed=seed).astype(np.float32)).to(dev)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)
    cbd = t(cb)
    zero = torch.zeros((n, n // 128), dtype=torch.int16, device=dev)
    m0 = SphqMatrix(n, n, bits, cbd, zero, zero)
    sg, ix, rc, sc, of = m0.encode(w)
    del w
    mats = [m0]
    for _ in range(P - 1):
        m = SphqMatrix(n, n, bits, cbd, sc, of)
        m.pack(sg, ix, rc)
        mats.append(m)
    torch.cuda.synchronize()
    return mats, t(x).view(torch.float16), x


def capture(mats, xd, ys, stream):
    import torch
    with torch.cuda.stream(stream):
        for m, y in zip(mats, ys):
            m.gemv_ptr(xd.data_ptr(), y.data_ptr(), 1, stream.cuda_stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for m, y in zip(mats, ys):
            m.gemv_ptr(xd.data_ptr(), y.data_ptr(), 1, stream.cuda_stream)
    return g


def run_gpu(args, world, rank, local):
    import torch
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_24875_gb300 import load
    load()
    hbm_peak, peak_kind = measured_peaks()
    L2 = l2_bytes()
    stream = torch.cuda.Stream(device=dev)

    # --- pools for the square sweep ---
    shapes = []
    for sid, (bits, n) in enumerate(inp.SQUARE_SWEEP):
        probe_bytes = n * n * (8 + 7 * bits - 8 + 4) // 64 + (n * n // 128) * 4
        P = max(2, int(np.ceil(2 * L2 / probe_bytes)) + 1)
        if args.quick:
            P = 2
        mats, xd, x = make_encoded_pool(bits, n, P, inp.seed_for(1, sid), dev)
        ys = [torch.empty((1, n), dtype=torch.float16, device=dev) for _ in mats]
        g = capture(mats, xd, ys, stream)
        shapes.append(dict(name=f"W{bits} {n}x{n}", bits=bits, n=n, mats=mats, xd=xd, ys=ys,
                           graph=g, bytes=mats[0].bytes(1), P=P, launches=P))
    # --- the W2 and W3 decoder stacks ---
    stacks = [] if args.no_stack else [make_stack(args, bits, dev, stream) for bits in (2, 3)]
    parts = shapes + stacks
    torch.cuda.synchronize()

    def step(evs=None):
        for i, s in enumerate(parts):
            torch.cuda.nvtx.range_push(s["name"])   # NVTX ranges for timeline tools
            if evs is not None:
                evs[i][0].record(stream)
            s["graph"].replay()
            if evs is not None:
                evs[i][1].record(stream)
            torch.cuda.nvtx.range_pop()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()

    K = args.steps
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in parts]
          for _ in range(K)]
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    dist_barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        h0 = time.perf_counter()
        with torch.cuda.stream(stream):
            t0.record(stream)
            for k in range(K):
                step(ev[k])
            t1.record(stream)
        torch.cuda.synchronize()
        clk.mark(h0, time.perf_counter())
    dist_barrier(world)
    total_ms = t0.elapsed_time(t1)
    total_ms = dist_max(world, total_ms)
    part_ms = [sum(ev[k][i][0].elapsed_time(ev[k][i][1]) for k in range(K))
               for i in range(len(parts))]
    launches = sum(s["launches"] for s in parts) * K
    step_bytes = sum(s["P"] * s["bytes"] for s in parts)
    value = step_bytes * K * world / (total_ms * 1e-3) / 1e9

    sweep = {}
    for s, ms in zip(shapes, part_ms):
        us = ms * 1e3 / (K * s["P"])
        gbs = s["bytes"] / (us * 1e-6) / 1e9
        sweep[s["name"]] = {"us_per_gemv": round(us, 3), "GB/s": round(gbs, 1),
                            "hbm_frac": round(gbs / hbm_peak, 4), "bytes": s["bytes"],
                            "pool": s["P"]}
    stack = {}
    for s, ms in zip(stacks, part_ms[len(shapes):]):
        us = ms * 1e3 / K
        gbs = s["bytes"] / (us * 1e-6) / 1e9
        stack[s["name"]] = {"us_per_token": round(us, 2), "layers": s["layers"], "gemvs": s["launches"],
                            "bytes_per_token": s["bytes"], "GB/s": round(gbs, 1),
                            "hbm_frac": round(gbs / hbm_peak, 4)}
    # dominant kernel: the instantiation (W2 or W3, batch 1) with the most
    # device time per step, over all its launches in the step
    per_bits = {}
    for s, ms in zip(parts, part_ms):
        b = per_bits.setdefault(s["bits"], [0.0, 0, 0])
        b[0] += ms
        b[1] += s["P"] * s["bytes"]
        b[2] += s["launches"]
    dom_bits = max(per_bits, key=lambda b: per_bits[b][0])
    d_ms, d_bytes, d_launches = per_bits[dom_bits]
    achieved = d_bytes * K / (d_ms * 1e-3) / 1e9
    traffic = None
    if kernel_digest() == TRAFFIC_DIGEST:
        traffic = round(TRAFFIC_RATIO[dom_bits] * d_bytes / d_launches)
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm_peak,
                "unit": "GB/s", "frac": round(achieved / hbm_peak, 4),
                "traffic": traffic,
                "kernel": f"gemv_kernel W{dom_bits} batch 1 ({d_launches} launches/step, "
                          f"{round(100 * d_ms / sum(part_ms), 1)}% of step device time)",
                "bytes_per_launch": round(d_bytes / d_launches),
                "us_per_launch": round(d_ms * 1e3 / (K * d_launches), 3),
                "peak_kind": peak_kind}

    # --- end to end through the host-buffer entry point ---
    e2e = run_e2e(args, shapes, stream)

    # --- the stacks with q|k|v and gate|up fused (4 GEMVs per layer) ---
    stack_fused = None if args.no_stack else run_fused_stacks(args, dev, stream, hbm_peak)

    for s in parts:
        for m in s["mats"]:
            m.close()
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": K, "warmup": args.warmup, "ms_per_step": round(total_ms / K, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "fp16 in, fp32 accumulate (2.25/3.125-bit codes)", "data": "synthetic",
        "config": {"workload": WORKLOAD,
                   "pools": {s["name"]: s["P"] for s in shapes},
                   "l2_policy": "inputs larger than L2: each pool > 2x L2 and each stack "
                                "> 10x L2, distinct buffers per GEMV",
                   "parallelism": f"replicas x{world}"},
        "hbm_frac": round(value / hbm_peak, 4),
        "sweep": sweep, "stack": stack or None, "stack_fused": stack_fused,
        "roofline": roofline, "e2e": e2e,
        "gpu_launches": launches,
    }
    return out, clk.summary()


def run_e2e(args, shapes, stream):
    import torch
    K = max(1, min(args.steps, 50))
    xs = [torch.empty((1, s["n"]), dtype=torch.float16).pin_memory() for s in shapes]
    ys = [torch.empty((1, s["n"]), dtype=torch.float16).pin_memory() for s in shapes]
    for xh, s in zip(xs, shapes):
        xh.copy_(s["xd"].cpu())
    for _ in range(3):
        for i, s in enumerate(shapes):
            s["mats"][0].gemv_host(xs[i], ys[i], stream=stream)
    stream.synchronize()
    t0 = time.perf_counter()
    for k in range(K):
        for i, s in enumerate(shapes):
            s["mats"][k % s["P"]].gemv_host(xs[i], ys[i], stream=stream)
        stream.synchronize()
    dt = time.perf_counter() - t0
    b = sum(s["bytes"] for s in shapes)
    return {"value": round(b * K / dt / 1e9, 1), "unit": UNIT,
            "h2d_bytes_per_step": sum(2 * s["n"] for s in shapes),
            "d2h_bytes_per_step": sum(2 * s["n"] for s in shapes),
            "us_per_step": round(dt / K * 1e6, 2)}


def run_fused_stacks(args, dev, stream, hbm_peak):
    """us/token of the W2 and W3 stacks with fused projections (CUDA events
    around each graph replay, after 3 warm-up replays)."""
    import torch
    res = {}
    for bits in (2, 3):
        st = make_stack(args, bits, dev, stream, fused=True)
        with torch.cuda.stream(stream):
            for _ in range(3):
                st["graph"].replay()
        torch.cuda.synchronize()
        reps = max(3, min(args.steps, 50))
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(reps):
                st["graph"].replay()
            e1.record(stream)
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / reps
        gbs = st["bytes"] / (us * 1e-6) / 1e9
        res[st["name"]] = {"us_per_token": round(us, 2), "layers": st["layers"],
                           "gemvs": st["launches"], "bytes_per_token": st["bytes"],
                           "GB/s": round(gbs, 1), "hbm_frac": round(gbs / hbm_peak, 4)}
        for m in st["mats"]:
            m.close()
        del st
        torch.cuda.empty_cache()
    return res


def make_stack(args, bits, dev, stream, fused=False):
    """The 28-layer linear stack at `bits`, as one CUDA graph of its GEMVs in
    layer order (one distinct packed matrix each): 7 per layer, or 4 with
    q|k|v and gate|up fused by row concatenation."""
    import torch

    from paper_2609_24875_gb300 import SphqMatrix
    layers = 2 if args.quick else inp.DECODER_LAYERS
    proj = inp.DECODER_PROJ_FUSED if fused else inp.DECODER_PROJ
    mats, ys, xs = [], [], []
    for i, (name, rows, cols) in enumerate(proj):
        codes, x = inp.random_codes(bits, rows, cols, seed=inp.seed_for(4, 10 * bits + i))
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)
        cb, sc, of = t(codes.codebook), t(codes.scale), t(codes.offset)
        sg, ix, rc = t(codes.sign), t(codes.idx), t(codes.rcode)
        xd = t(x).view(torch.float16)
        for l in range(layers):
            m = SphqMatrix(rows, cols, bits, cb, sc, of)
            m.pack(sg, ix, rc)
            mats.append((l, i, m))
            xs.append(xd)
            ys.append(torch.empty((1, rows), dtype=torch.float16, device=dev))
        del sg, ix, rc
    order = sorted(range(len(mats)), key=lambda j: (mats[j][0], mats[j][1]))
    seq = [(mats[j][2], xs[j], ys[j]) for j in order]
    with torch.cuda.stream(stream):
        for m, xd, yd in seq:
            m.gemv_ptr(xd.data_ptr(), yd.data_ptr(), 1, stream.cuda_stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for m, xd, yd in seq:
            m.gemv_ptr(xd.data_ptr(), yd.data_ptr(), 1, stream.cuda_stream)
    return dict(name=f"W{bits}" + (" fused" if fused else ""), bits=bits, graph=g,
                mats=[m for m, _, _ in seq], keep=(xs, ys), layers=layers,
                bytes=sum(m.bytes(1) for m, _, _ in seq), P=1, launches=len(seq))


# ---------------------------------------------------------------------------
# CPU oracle (cpu_baseline leg and --impl reference)
# ---------------------------------------------------------------------------

def oracle_sample(seconds: float, threads: int):
    """Times the float64 oracle (decode + matvec, row by row) on row samples of
    the step's matrices -- the sweep's four shapes and the W2 / W3 decoder
    projections of the stack -- until about `seconds` have elapsed.  Returns
    (GB/s over the sampled rows' share of the algorithmic bytes, description)."""
    import oracle
    oracle.set_threads(threads)
    per_shape = []
    for sid, (bits, n) in enumerate(inp.SQUARE_SWEEP):
        codes, x = inp.random_codes(bits, 64, n, seed=inp.seed_for(1, sid))
        per_shape.append((bits, n, n, codes, x))
    for bits in (2, 3):
        for i, (_, rows, cols) in enumerate(inp.DECODER_PROJ):
            codes, x = inp.random_codes(bits, 32, cols, seed=inp.seed_for(4, 10 * bits + i))
            per_shape.append((bits, rows, cols, codes, x))
    done_bytes, t_total, rows_done = 0.0, 0.0, 0
    budget = seconds / len(per_shape)
    for bits, rows, cols, codes, x in per_shape:
        full_bytes = (rows * cols * (7 * bits + 4) / 64 + rows * cols / 128 * 4
                      + (1 << (7 * bits - 8)) * 16 + 2 * (rows + cols))
        t0 = time.perf_counter()
        while True:
            oracle.decode_gemv(codes.codebook, codes.scale, codes.offset, codes.sign,
                               codes.idx, codes.rcode, x)
            rows_done += codes.rows
            done_bytes += full_bytes * codes.rows / rows
            if time.perf_counter() - t0 > budget:
                break
        t_total += time.perf_counter() - t0
    gbs = done_bytes / t_total / 1e9
    desc = (f"float64 oracle decode+matvec on row samples (64 / 32 rows) of the W2/W3 4096^2 and "
            f"8192^2 matrices and the W2/W3 decoder projections, {rows_done} rows in "
            f"{t_total:.1f} s, bytes scaled to the rows' share")
    return gbs, desc, t_total


def run_reference(args, world, rank):
    if rank != 0:
        return None
    import oracle
    threads = oracle.max_threads()
    vals = []
    for _ in range(args.warmup):
        oracle_sample(0.2, threads)
    t0 = time.perf_counter()
    per = max(0.5, min(10.0, 60.0 / max(1, args.steps)))
    for _ in range(args.steps):
        v, desc, _ = oracle_sample(per, threads)
        vals.append(v)
    dt = time.perf_counter() - t0
    value = statistics.median(vals)
    hbm_peak, _ = measured_peaks()
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 2), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "parallelism": "cpu oracle"},
        "hbm_frac": round(value / hbm_peak, 6),
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": threads,
                         "kind": "oracle", "sample": desc},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def run_case(spec: str, pool: int, launches: int):
    """Profiling driver: `bits:n[:batch]` or `bits:RxC[:batch]` -> `pool`
    distinct packed n x n (R x C) matrices, `launches` GEMVs round robin on one
    stream, no timing (for running under ncu).  bits `3v3` selects W3 with
    3-bit radius codes, `dDvV` the 8/D/V split (e.g. `d7v2`), `v4` / `v16` 4-D
    / 16-D vectors (Tab. 7, W2 allocation); a leading `e` (`e3:8192`) packs the
    encoded configuration's codes (sphq_encode on the Gaussian weights of the
    square sweep, batch 1) instead of random codes."""
    import torch

    head, size, *rest = spec.split(":")
    encoded = head.startswith("e")
    vdim = {"v4": 4, "v16": 16}.get(head, 8)
    bits, vbits, K = (2, 4, 1 << (2 * (vdim - 1) - vdim)) if vdim != 8 else parse_split(head.lstrip("e"))
    rows, n = (int(v) for v in size.split("x")) if "x" in size else (int(size), int(size))
    batch = int(rest[0]) if rest else 1
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2609_24875_gb300 import SphqMatrix
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)
    if encoded:
        if rows != n or batch != 1 or (bits, n) not in inp.SQUARE_SWEEP:
            raise SystemExit("--case e...: one of the square sweep's shapes, batch 1")
        mats, xd, _ = make_encoded_pool(bits, n, pool,
                                        inp.seed_for(1, inp.SQUARE_SWEEP.index((bits, n))), dev)
    else:
        if vdim != 8:
            codes, x = inp.random_codes_dim(vdim, 2, rows, n, seed=1, B=batch)
        else:
            codes, x = inp.random_codes(bits, rows, n, seed=1, B=batch, radius_bits=vbits, K=K)
        mats = []
        for _ in range(pool):
            m = SphqMatrix(rows, n, bits, t(codes.codebook), t(codes.scale), t(codes.offset),
                           radius_bits=vbits, K=K, dim=vdim)
            m.pack(t(codes.sign.astype(np.uint8) if vdim == 4 else codes.sign), t(codes.idx),
                   t(codes.rcode))
            mats.append(m)
        xd = t(x).view(torch.float16)
    ys = [torch.empty((batch, rows), dtype=torch.float16, device=dev) for _ in mats]
    s = torch.cuda.current_stream()
    for i in range(launches):
        mats[i % pool].gemv_ptr(xd.data_ptr(), ys[i % pool].data_ptr(), batch, s.cuda_stream)
    torch.cuda.synchronize()
    print(f"case W{bits} V={vbits} {rows}x{n} batch {batch}: {launches} launches over {pool} "
          "matrices done")


def parse_split(head: str):
    """bits token of the profiling drivers -> (bits, radius bits, K): "2", "3",
    "3v3" (W3, 3-bit radius codes) or "2:D:V" style "d7v2" (8/7/2)."""
    if head == "3v3":
        return 3, 3, 8192
    if head.startswith("d"):
        d, v = head[1:].split("v")
        return 2, int(v), 1 << int(d)
    b = int(head)
    return b, 4, 1 << (7 * b - 8)


def run_gemm_case(spec: str, launches: int):
    """Profiling driver of the prefill GEMM: `bits:rows:cols:batch[:ws]` ->
    `launches` sphq_gemm calls on one matrix (with `:ws`, sphq_gemm_ws calls:
    the decode pass and the dense pass), no timing (for ncu)."""
    import torch

    head, *rest = spec.split(":")
    two_pass = rest[-1] == "ws"
    if two_pass:
        rest = rest[:-1]
    bits, vbits, K = parse_split(head)
    rows, cols, batch = (int(v) for v in rest)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2609_24875_gb300 import SphqMatrix
    codes, x = inp.random_codes(bits, rows, cols, seed=1, B=batch, radius_bits=vbits, K=K)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)
    m = SphqMatrix(rows, cols, bits, t(codes.codebook), t(codes.scale), t(codes.offset),
                   radius_bits=vbits, K=K)
    m.pack(t(codes.sign), t(codes.idx), t(codes.rcode))
    xd = t(x).view(torch.float16)
    y = torch.empty((batch, rows), dtype=torch.float16, device=dev)
    s = torch.cuda.current_stream()
    ws = torch.empty(rows * cols, dtype=torch.float16, device=dev) if two_pass else None
    for _ in range(launches):
        if two_pass:
            m.gemm_ws(xd, ws, y=y)
        else:
            m.gemm_ptr(xd.data_ptr(), y.data_ptr(), batch, s.cuda_stream)
    m.check()
    print(f"gemm case W{bits} V={vbits} K={K} {rows}x{cols} batch {batch}"
          f"{' two-pass' if two_pass else ''}: {launches} launches done")


def run_encode_case(spec: str, launches: int):
    """Profiling driver of the encoder: `bits:rows:cols` (bits token as for
    --case) -> `launches` sphq_encode calls on N(0, 0.02^2) weights, no timing."""
    import torch

    head, *rest = spec.split(":")
    bits, vbits, K = parse_split(head)
    rows, cols = (int(v) for v in rest)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2609_24875_gb300 import SphqMatrix
    cb = inp.make_codebook(np.random.Generator(np.random.PCG64(1)), K)
    ones = inp.to_f16_bits(np.ones((rows, cols // 128)))
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16))).to(dev)
    m = SphqMatrix(rows, cols, bits, t(cb), t(ones), t(ones), radius_bits=vbits, K=K)
    w = torch.from_numpy(inp.gaussian_weights(rows, cols, seed=1).astype(np.float32)).to(dev)
    for _ in range(launches):
        m.encode(w)
    torch.cuda.synchronize()
    print(f"encode case W{bits} V={vbits} K={K} {rows}x{cols}: {launches} calls done")


def encode_report():
    """GPU encoder (sphq_encode) throughput on N(0, 0.02^2) weights: ms per
    matrix (min of 3 calls after one warm-up, host clock around a synchronous
    call), 8-D vectors and coarse scores per second, and the tensor-core share
    (two passes of one 128 x 256 x 16 MMA per 256 entries); the single-
    precision CPU oracle encoder on a 64-row sample for comparison."""
    import torch

    import oracle
    from paper_2609_24875_gb300 import SphqMatrix
    dev = torch.device("cuda", 0)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16))).to(dev)
    out = {}
    for name, (bits, v, K) in (("W2", (2, 4, 64)), ("8/8/2", (2, 2, 256)), ("W3", (3, 4, 8192))):
        cb = inp.make_codebook(np.random.Generator(np.random.PCG64(1)), K)
        for n in (4096, 8192):
            ones = inp.to_f16_bits(np.ones((n, n // 128)))
            m = SphqMatrix(n, n, bits, t(cb), t(ones), t(ones), radius_bits=v, K=K)
            w = (torch.randn(n, n, device=dev) * 0.02).float()
            m.encode(w)
            torch.cuda.synchronize()
            ts = []
            for _ in range(3):
                t0 = time.perf_counter()
                m.encode(w)
                torch.cuda.synchronize()
                ts.append(time.perf_counter() - t0)
            ms = min(ts) * 1e3
            nv = n * n / 8
            out[f"{name} {n}x{n}"] = {"ms": round(ms, 3), "Gvec/s": round(nv / ms / 1e6, 3),
                                      "Tscores/s": round(nv * K / ms / 1e9, 3)}
            m.close()
            del w
            torch.cuda.empty_cache()
        wc = inp.gaussian_weights(64, 4096, seed=2).astype(np.float32)
        oracle.set_threads(oracle.max_threads())
        t0 = time.perf_counter()
        oracle.encode_fp32(wc, cb, v)
        cpu_s = time.perf_counter() - t0
        out[f"{name} cpu_oracle_fp32"] = {"Gvec/s": round(64 * 512 / cpu_s / 1e9, 6),
                                          "threads": oracle.max_threads()}
    return out


def gemm_report(hbm_peak):
    """Prefill GEMM (sphq_gemm) against the tensor-core roofline: TFLOP/s =
    2 * batch * rows * cols / time (median of 10 timed calls after warm-up,
    events on the launching stream), fraction of the measured bf16 dense peak
    (fp16 runs at the bf16 rate); a dense fp16 cuBLAS GEMM on the decoded
    weights of the same shape is timed beside it as context."""
    import torch

    from paper_2609_24875_gb300 import SphqMatrix
    dev = torch.device("cuda", 0)
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    tf_peak = float(peaks.get("bf16_tflops", 1900.0))
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)
    stream = torch.cuda.Stream(device=dev)

    def timed(fn, reps=10):
        with torch.cuda.stream(stream):
            for _ in range(3):
                fn()
        stream.synchronize()
        times = []
        for _ in range(reps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                e0.record(stream)
                fn()
                e1.record(stream)
            stream.synchronize()
            times.append(e0.elapsed_time(e1) * 1e3)
        return statistics.median(times)

    out = {"peak_tflops": tf_peak}
    for name, (bits, v, K) in (("W2", (2, 4, 64)), ("W3", (3, 4, 8192)), ("W3V3", (3, 3, 8192)),
                               ("8/8/2", (2, 2, 256))):
        for rows, cols, batch in ((3584, 3584, 512), (18944, 3584, 2048), (8192, 8192, 4096)):
            codes, _ = inp.random_codes(bits, rows, cols, seed=inp.seed_for(5, rows % 97),
                                        radius_bits=v, K=K)
            m = SphqMatrix(rows, cols, bits, t(codes.codebook), t(codes.scale), t(codes.offset),
                           radius_bits=v, K=K)
            m.pack(t(codes.sign), t(codes.idx), t(codes.rcode))
            x = torch.randn(batch, cols, device=dev).half()
            y = torch.empty(batch, rows, device=dev, dtype=torch.half)
            us = timed(lambda: m.gemm_ptr(x.data_ptr(), y.data_ptr(), batch, stream.cuda_stream))
            m.check(stream)
            # the two-pass form (W_hat decoded into a workspace, then the dense
            # tensor-core pass), whichever the library would choose
            ws = torch.empty(rows * cols, dtype=torch.float16, device=dev)
            us_2 = timed(lambda: m.gemm_ws(x, ws, y=y, stream=stream))
            m.check(stream)
            advice = m.gemm_workspace(batch)
            del ws
            wd = m.decode()
            torch.cuda.synchronize()
            us_d = timed(lambda: torch.matmul(x, wd.t()))
            fl = 2.0 * batch * rows * cols
            best = min(us, us_2)
            out[f"{name} {rows}x{cols} B{batch}"] = {
                "us": round(us, 2), "TF/s": round(fl / us / 1e6, 1),
                "tensor_frac": round(fl / us / 1e6 / tf_peak, 4),
                "two_pass_us": round(us_2, 2), "two_pass_TF/s": round(fl / us_2 / 1e6, 1),
                "library_choice": "two-pass" if advice else "fused",
                "best_tensor_frac": round(fl / best / 1e6 / tf_peak, 4),
                "dense_fp16_cublas_us": round(us_d, 2)}
            m.close()
            del wd, x, y
            torch.cuda.empty_cache()
    return out


def midbatch_report():
    """Batches of 16-256 rows: sphq_gemm (GEMV launches of up to 16 rows or the
    tensor-core kernel, whichever the library picks) against sphq_gemm_ws with
    the workspace sphq_gemm_workspace advises (the split-K form where it
    applies); one call after writing a 256 MiB buffer (an L2 flush), CUDA
    events around the call, median of 15."""
    import torch

    from paper_2609_24875_gb300 import SphqMatrix
    dev = torch.device("cuda", 0)
    stream = torch.cuda.Stream(device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)

    def timed(fn, reps=15):
        with torch.cuda.stream(stream):
            for _ in range(3):
                fn()
        stream.synchronize()
        times = []
        for _ in range(reps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                flush.zero_()
                e0.record(stream)
                fn()
                e1.record(stream)
            stream.synchronize()
            times.append(e0.elapsed_time(e1) * 1e3)
        return statistics.median(times)

    out = {}
    for bits in (2, 3):
        for rows, cols in ((8192, 8192), (3584, 18944)):
            codes, _ = inp.random_codes(bits, rows, cols, seed=inp.seed_for(6, rows % 97))
            m = SphqMatrix(rows, cols, bits, t(codes.codebook), t(codes.scale), t(codes.offset))
            m.pack(t(codes.sign), t(codes.idx), t(codes.rcode))
            for batch in (16, 32, 64, 128, 256):
                x = torch.randn(batch, cols, device=dev).half()
                y = torch.empty(batch, rows, device=dev, dtype=torch.half)
                us = timed(lambda: m.gemm_ptr(x.data_ptr(), y.data_ptr(), batch, stream.cuda_stream))
                e = {"gemm_us": round(us, 2), "ksplit": m.gemm_shape(batch)["ksplit"]}
                need = m.gemm_workspace(batch)
                if need:
                    ws = torch.empty(need, dtype=torch.uint8, device=dev)
                    e["ws_us"] = round(timed(lambda: m.gemm_ws(x, ws, y=y, stream=stream)), 2)
                    e["ws_bytes"] = need
                    del ws
                m.check(stream)
                out[f"W{bits} {rows}x{cols} B{batch}"] = e
            m.close()
            torch.cuda.empty_cache()
    del flush
    torch.cuda.empty_cache()
    return out


def study_gather16(mode: int, iters: int = 4096) -> float:
    """Random 32-byte reads per second from a 512 KiB table (0: L2, 1: cluster
    shared memory, 2: local shared memory), from the profiling library
    libsphq_study.so (built next to libsphq.so, not part of its C ABI)."""
    import ctypes
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2609_24875_gb300", "libsphq_study.so"))
    lib.sphq_study_gather16.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_double)]
    lib.sphq_study_gather16.restype = ctypes.c_int
    rate = ctypes.c_double()
    rc = lib.sphq_study_gather16(mode, iters, ctypes.byref(rate))
    if rc != 0:
        raise RuntimeError(f"sphq_study_gather16 failed ({rc})")
    return rate.value


def steady_us(mats, xd, ys, batch, stream, reps=20):
    """Median over `reps` graph replays of the mean time per GEMV of a CUDA
    graph of back-to-back launches over the pool."""
    import torch
    with torch.cuda.stream(stream):
        for m, y in zip(mats, ys):
            m.gemv_ptr(xd.data_ptr(), y.data_ptr(), batch, stream.cuda_stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for m, y in zip(mats, ys):
            m.gemv_ptr(xd.data_ptr(), y.data_ptr(), batch, stream.cuda_stream)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    times = []
    for _ in range(reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            g.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1) * 1e3 / len(mats))
    del g
    return statistics.median(times)


def cold_us(m, xd, y, batch, stream, flush, reps=10):
    """Isolated call: L2 flushed by writing a buffer of twice its size, then
    one GEMV timed alone with events (median of `reps`)."""
    import torch
    times = []
    for _ in range(reps):
        with torch.cuda.stream(stream):
            flush.fill_(1.0)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            m.gemv_ptr(xd.data_ptr(), y.data_ptr(), batch, stream.cuda_stream)
            e1.record(stream)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1) * 1e3)
    return statistics.median(times)


def run_report(args):
    """Per-configuration table (steady state, isolated cold calls, small
    batch, 7B-class projections, CPU oracle) printed as one JSON object.
    Supplementary to the contract line; not part of the timed step."""
    import torch

    from paper_2609_24875_gb300 import SphqMatrix
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(device=dev)
    hbm_peak, _ = measured_peaks()
    L2 = l2_bytes()
    flush = torch.empty(2 * L2 // 4, dtype=torch.float32, device=dev)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).to(dev)

    def pool_for(bits, rows, cols, seed, batch, vbits=4, K=None):
        codes, x = inp.random_codes(bits, rows, cols, seed=seed, B=batch, radius_bits=vbits, K=K)
        one = (8 + int(np.log2(codes.K)) + vbits) * rows * cols // 64
        P = min(512, max(2, int(np.ceil(2 * L2 / one)) + 1))
        cb, sc, of = t(codes.codebook), t(codes.scale), t(codes.offset)
        sg, ix, rc = t(codes.sign), t(codes.idx), t(codes.rcode)
        mats = []
        for _ in range(P):
            m = SphqMatrix(rows, cols, bits, cb, sc, of, radius_bits=vbits, K=codes.K)
            m.pack(sg, ix, rc)
            mats.append(m)
        xd = t(x).view(torch.float16)
        ys = [torch.empty((batch, rows), dtype=torch.float16, device=dev) for _ in mats]
        return mats, xd, ys

    def entry(bits, rows, cols, seed, batch, cold=False, vbits=4, K=None):
        mats, xd, ys = pool_for(bits, rows, cols, seed, batch, vbits, K)
        b = mats[0].bytes(batch)
        us = steady_us(mats, xd, ys, batch, stream)
        e = {"us": round(us, 3), "GB/s": round(b / us / 1e3, 1),
             "hbm_frac": round(b / us / 1e3 / hbm_peak, 4), "bytes": b, "pool": len(mats)}
        if cold:
            cu = cold_us(mats[0], xd, ys[0], batch, stream, flush)
            e["cold_us"] = round(cu, 3)
            # the same graph of back-to-back launches without programmatic
            # dependent launch (each GEMV waits for the previous to finish)
            for m in mats:
                m.set_pdl(False)
            e["us_no_pdl"] = round(steady_us(mats, xd, ys, batch, stream), 3)
        for m in mats:
            m.close()
        torch.cuda.empty_cache()
        return e

    def entry_encoded(bits, n, seed):
        one = (7 * bits + 4) * n * n // 64
        P = min(512, max(2, int(np.ceil(2 * L2 / one)) + 1))
        mats, xd, _ = make_encoded_pool(bits, n, P, seed, dev)
        ys = [torch.empty((1, n), dtype=torch.float16, device=dev) for _ in mats]
        b = mats[0].bytes(1)
        us = steady_us(mats, xd, ys, 1, stream)
        e = {"us": round(us, 3), "GB/s": round(b / us / 1e3, 1),
             "hbm_frac": round(b / us / 1e3 / hbm_peak, 4), "bytes": b, "pool": P,
             "codes": "GPU encoder on Gaussian weights with outliers"}
        e["cold_us"] = round(cold_us(mats[0], xd, ys[0], 1, stream, flush), 3)
        for m in mats:
            m.set_pdl(False)
        e["us_no_pdl"] = round(steady_us(mats, xd, ys, 1, stream), 3)
        for m in mats:
            m.close()
        torch.cuda.empty_cache()
        return e

    rep = {"steady": "median of 20 graph replays over a pool > 2x L2, back-to-back with PDL",
           "cold": "one call after writing a 2x L2 buffer, events around the call",
           "us_no_pdl": "steady state with plain stream-ordered launches (sphq_set_pdl 0)"}
    rep["cfg0_w2_1024"] = entry(2, 1024, 1024, inp.seed_for(0, 0), 1, cold=True)
    rep["cfg1_sweep"] = {f"W{b} {n}x{n}": entry_encoded(b, n, inp.seed_for(1, i))
                         for i, (b, n) in enumerate(inp.SQUARE_SWEEP)}
    # the same shapes on uniformly random codes: the codebook's bank
    # conflicts depend on the index distribution, the bytes do not
    rep["cfg1_random_codes"] = {f"W{b} {n}x{n}": entry(b, n, n, inp.seed_for(1, i), 1)
                                for i, (b, n) in enumerate(inp.SQUARE_SWEEP)}
    rep["cfg2_w2_proj"] = {f"{nm} {r}x{c}": entry(2, r, c, inp.seed_for(2, i), 1)
                           for i, (nm, r, c) in enumerate(inp.DECODER_PROJ) if nm not in ("v", "up")}
    rep["cfg3_w3_proj_batch"] = {f"{nm} {r}x{c} B{bt}": entry(3, r, c, inp.seed_for(3, i), bt)
                                 for i, (nm, r, c) in enumerate(inp.DECODER_PROJ)
                                 if nm in ("q", "k", "gate", "down") for bt in (1, 2, 4, 8, 16)}
    # Compute rooflines of the small-batch GEMV beside HBM: the mma.sync rate
    # the kernel issues its products to (one m16n8k16 per 8 cycles per SM
    # sub-partition, measured on this part; 8 per 256-vector unit, 16 for
    # 9-16 rows, whose two batch halves each take the decoded block) and the
    # plain FP32 FMA rate (128 per SM per cycle, 2 flops each), at the SM
    # clock sampled meanwhile.
    mhz = sm_clock_mhz()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    mma_peak = sms * 4 / 8 * mhz * 1e6
    alu_peak = sms * 128 * 2 * mhz * 1e6
    for key, e in rep["cfg3_w3_proj_batch"].items():
        rc_ = key.split()[1].split("x")
        r, c, bt = int(rc_[0]), int(rc_[1]), int(key.split("B")[-1])
        mma = (16 if bt > 8 else 8) * ((r + 15) // 16) * (c // 128)
        e["mma_frac"] = round(mma / (e["us"] * 1e-6) / mma_peak, 4)
        e["fp32_alu_frac"] = round(2.0 * bt * r * c / (e["us"] * 1e-6) / alu_peak, 4)
        fr = {"hbm": e["hbm_frac"], "mma": e["mma_frac"], "fp32_alu": e["fp32_alu_frac"]}
        e["nearest_roofline"] = max(fr, key=fr.get)
    rep["compute_rooflines"] = {"sm_mhz": mhz, "mma_sync_per_s": mma_peak,
                                "fp32_flops_per_s": alu_peak}
    # general bit splits: W3 with 3-bit radius codes (3.00 bits per weight) and
    # the small-codebook splits of the bit-allocation ablation (sign/index/radius)
    rep["w3v3_square"] = {f"W3V3 {n}x{n} B{bt}": entry(3, n, n, inp.seed_for(1, 10 + i), bt,
                                                       cold=bt == 1, vbits=3)
                          for i, n in enumerate((4096, 8192)) for bt in (1, 4)}
    rep["tab4_splits_8192"] = {f"8/{d}/{v} 8192x8192 B1": entry(2, 8192, 8192,
                                                               inp.seed_for(1, 20 + 10 * d + v),
                                                               1, vbits=v, K=1 << d)
                               for d, v in ((6, 2), (6, 3), (7, 2), (7, 3), (8, 2), (6, 4))}
    # 4-D vectors (the vector-dimension comparison at the W2 allocation)
    rep["dim4"] = {}
    for i, n in enumerate((4096, 8192)):
        for bt in (1, 4):
            codes, x = inp.random_codes_dim(4, 2, n, n, seed=inp.seed_for(1, 30 + i), B=bt)
            one = n * n * 10 // 32
            P = min(512, max(2, int(np.ceil(2 * L2 / one)) + 1))
            cb, sc, of = t(codes.codebook), t(codes.scale), t(codes.offset)
            sg, ix, rc = t(codes.sign.astype(np.uint8)), t(codes.idx), t(codes.rcode)
            mats = []
            for _ in range(P):
                m = SphqMatrix(n, n, 2, cb, sc, of, radius_bits=4, K=4, dim=4)
                m.pack(sg, ix, rc)
                mats.append(m)
            xd = t(x).view(torch.float16)
            ys = [torch.empty((bt, n), dtype=torch.float16, device=dev) for _ in mats]
            b = mats[0].bytes(bt)
            us = steady_us(mats, xd, ys, bt, stream)
            rep["dim4"][f"4-D {n}x{n} B{bt}"] = {
                "us": round(us, 3), "GB/s": round(b / us / 1e3, 1),
                "hbm_frac": round(b / us / 1e3 / hbm_peak, 4), "bytes": b, "pool": P}
            for m in mats:
                m.close()
            torch.cuda.empty_cache()
    # 16-D study: random 32-byte entry reads from a 512 KiB codebook
    rates = {name: study_gather16(mode) for mode, name in
             ((0, "l2"), (1, "cluster_dsmem_4"), (2, "local_smem"))}
    # 16-D W2 payload per vector: 16 sign + 14 index + 4 radius bits + params
    need = hbm_peak * 1e9 / (34 / 8 + 4 * 16 / 128)
    rep["gather16_study"] = {k: {"G_entries/s": round(v / 1e9, 1),
                                 "max_hbm_frac_16d": round(min(1.0, v / need), 3)}
                             for k, v in rates.items()}
    # 16-D vectors: the GEMV gathers one 32-byte codebook entry per vector
    # through L1/L2, so beside HBM its roofline is the L2 gather rate above
    rep["dim16"] = {}
    for i, (r, c) in enumerate(((4096, 4096), (8192, 8192), (3584, 18944))):
        for bt in (1, 8):
            codes, x = inp.random_codes_dim(16, 2, r, c, seed=inp.seed_for(1, 40 + i), B=bt)
            one = r * c * 19 // 64
            P = min(512, max(2, int(np.ceil(2 * L2 / one)) + 1))
            cb, sc, of = t(codes.codebook), t(codes.scale), t(codes.offset)
            sg, ix, rc = t(codes.sign), t(codes.idx), t(codes.rcode)
            mats = []
            for _ in range(P):
                m = SphqMatrix(r, c, 2, cb, sc, of, radius_bits=4, K=1 << 14, dim=16)
                m.pack(sg, ix, rc)
                mats.append(m)
            xd = t(x).view(torch.float16)
            ys = [torch.empty((bt, r), dtype=torch.float16, device=dev) for _ in mats]
            b = mats[0].bytes(bt)
            us = steady_us(mats, xd, ys, bt, stream)
            ents = r * c // 16 / us / 1e3  # G entries gathered per second
            rep["dim16"][f"16-D {r}x{c} B{bt}"] = {
                "us": round(us, 3), "GB/s": round(b / us / 1e3, 1),
                "hbm_frac": round(b / us / 1e3 / hbm_peak, 4), "G_entries/s": round(ents, 1),
                "l2_gather_frac": round(ents / (rates["l2"] / 1e9), 4), "bytes": b, "pool": P,
                "cluster_size": mats[0].plan(bt)["cluster_size"]}
            for m in mats:
                m.close()
            torch.cuda.empty_cache()
    rep["prefill_gemm"] = gemm_report(hbm_peak)
    rep["mid_batch_gemm"] = midbatch_report()
    rep["encode"] = encode_report()
    rep["oracle_timing"] = oracle_timing()
    print(json.dumps(rep), flush=True)


def sm_clock_mhz() -> float:
    """Current SM clock from nvidia-smi (the maximum if the query fails)."""
    try:
        out = subprocess.run(["nvidia-smi", "-i", "0", "--query-gpu=clocks.sm,clocks.max.sm",
                              "--format=csv,noheader,nounits"], capture_output=True, text=True,
                             timeout=10).stdout.strip().split(",")
        cur, mx = float(out[0]), float(out[1])
        return cur if cur > 0.5 * mx else mx
    except (OSError, ValueError, IndexError, subprocess.TimeoutExpired):
        return 2070.0


def oracle_timing(budget_s: float = 0.5):
    """The float64 CPU oracle (decode + matvec) per configuration, on one thread
    and on all host cores: us per GEMV for configurations 0-3 (every shape and
    batch) and us per token for configuration 4 (one decoder layer's seven
    GEMVs, times 28 layers).  Each GEMV is timed on a sample of its rows until
    `budget_s` elapses and scaled to the full row count (rows cost the same)."""
    import oracle

    def per_gemv(bits, rows, cols, batch, threads, seed):
        sample = min(rows, 256)
        codes, x = inp.random_codes(bits, sample, cols, seed=seed, B=batch)
        oracle.set_threads(threads)
        n, t0 = 0, time.perf_counter()
        while True:
            oracle.decode_gemv(codes.codebook, codes.scale, codes.offset, codes.sign,
                               codes.idx, codes.rcode, x)
            n += 1
            if time.perf_counter() - t0 > budget_s:
                break
        return (time.perf_counter() - t0) / n * rows / sample * 1e6

    allc = oracle.max_threads()
    out = {"cores": allc, "method": f"row samples of 256 rows, timed for {budget_s} s each, "
                                    "scaled to the full matrix; config 4 = one layer x 28"}
    cases = [("cfg0 W2 1024x1024 B1", 2, 1024, 1024, 1, inp.seed_for(0))]
    cases += [(f"cfg1 W{b} {n}x{n} B1", b, n, n, 1, inp.seed_for(1, i))
              for i, (b, n) in enumerate(inp.SQUARE_SWEEP)]
    cases += [(f"cfg2 W2 {nm} {r}x{c} B1", 2, r, c, 1, inp.seed_for(2, i))
              for i, (nm, r, c) in enumerate(inp.DECODER_PROJ)]
    cases += [(f"cfg3 W3 {nm} {r}x{c} B{bt}", 3, r, c, bt, inp.seed_for(3, i))
              for i, (nm, r, c) in enumerate(inp.DECODER_PROJ) for bt in (1, 2, 4, 8)]
    for name, b, r, c, bt, seed in cases:
        out[name] = {"us_1_thread": round(per_gemv(b, r, c, bt, 1, seed), 1),
                     f"us_{allc}_threads": round(per_gemv(b, r, c, bt, allc, seed), 1)}
    for bits in (2, 3):
        layer = {th: sum(per_gemv(bits, r, c, 1, th, inp.seed_for(4, 10 * bits + i))
                         for i, (_, r, c) in enumerate(inp.DECODER_PROJ)) for th in (1, allc)}
        out[f"cfg4 W{bits} stack us/token"] = {
            "us_1_thread": round(layer[1] * inp.DECODER_LAYERS, 1),
            f"us_{allc}_threads": round(layer[allc] * inp.DECODER_LAYERS, 1)}
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--quick", action="store_true", help="pools of 2 / 2 stack layers (smoke runs)")
    ap.add_argument("--no-stack", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--case", default="", help="profiling driver: bits:n[:batch] or bits:RxC[:batch], no timing")
    ap.add_argument("--pool", type=int, default=4, help="--case: distinct matrices")
    ap.add_argument("--launches", type=int, default=8, help="--case: GEMV launches")
    ap.add_argument("--gemm-case", default="",
                    help="prefill GEMM profiling driver: bits:rows:cols:batch, no timing")
    ap.add_argument("--encode-case", default="",
                    help="encoder profiling driver: bits:rows:cols, no timing")
    ap.add_argument("--report", action="store_true",
                    help="supplementary per-configuration table (one JSON object)")
    args = ap.parse_args()
    if args.case:
        run_case(args.case, args.pool, args.launches)
        return
    if args.gemm_case:
        run_gemm_case(args.gemm_case, args.launches)
        return
    if args.encode_case:
        run_encode_case(args.encode_case, args.launches)
        return
    if args.report:
        run_report(args)
        return
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world, rank, local = dist_setup()

    if args.impl == "reference":
        out = run_reference(args, world, rank)
        if rank == 0:
            print(json.dumps(out), flush=True)
        return

    out, clocks = run_gpu(args, world, rank, local)
    if rank == 0:
        out["clocks"] = clocks
        if world == 1 and not args.no_cpu_baseline:
            import oracle
            threads = oracle.max_threads()
            v, desc, _ = oracle_sample(args.cpu_seconds, threads)
            out["cpu_baseline"] = {"value": round(v, 4), "unit": UNIT, "cores": threads,
                                   "kind": "oracle", "sample": desc}
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
