#!/usr/bin/env python3
"""Benchmark of the FOVEA retrieve+fuse step on GB300.

One step = one fovea_retrieve_fuse call over a batch of draft states against a
visual memory built once beforehand (query LN + projection, scores over every
valid entry, cumulative-mass selection, readout, gated correction + RMSNorm).
Metric: draft states per second through retrieve+fuse (higher is better),
with the roofline fraction of the dominant kernel and of the whole step.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 2]
  python bench.py --impl reference ...   # the CPU oracle as the reference arm

Multi-GPU (torchrun, one rank per GPU): every rank runs an independent
replica of the workload (the path has no exchange step); value = the draft
states of all ranks / the slowest rank's time.
"""

from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import workloads  # noqa: E402

METRIC = "draft states/sec through retrieve+fuse at 1 GB300; % of HBM/tensor roofline"
UNIT = "draft_states/s"
L2_FLUSH_BYTES = 512 << 20
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {k: float(p[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained")}, "measured"
    except Exception:
        return dict(PEAKS_FALLBACK), "fallback"


# ---------------------------------------------------------------------------
# Algorithmic bytes / flops (what the method itself must move and compute)
# ---------------------------------------------------------------------------

def step_cost(w: workloads.Workload, counts: np.ndarray, indices: np.ndarray, projected: bool,
              folded: bool = False):
    """Per-step algorithmic bytes and flops: W_Q, the fusion weights, every
    valid key of every sequence, the unique selected memory rows, row I/O
    (h in, h_hat out, counts and indices); scores and hidden activations are
    intermediates and are not counted.  `projected`: the step reads the
    memory's projected values p_i = [W_f1 ; W_g1]_r u_i (2H wide) instead of
    the values, and only the h-half of the first fusion layer's weights.
    `folded`: the step scores x_h against the memory's folded keys
    W_Q^T k_i (formed with the memory, a hi / lo pair of bf16 values, so
    twice the key bytes), and W_Q is not read and q not formed."""
    d, H, N = w.d, w.params["b_f1"].shape[0], w.N
    es = 2 if w.dtype == "bf16" else 4
    fuse1 = 2 * H * (d if projected else 2 * d)
    weights = (0 if folded else d * d) + fuse1 + d * H + H + 2 * H + d + H + 1 + d   # W_Q, W_f1/W_g1, W_f2, biases, rms
    weights += 2 * d + 2 * d      # LN_h gamma/beta + the E_dep rows touched (bound: 2 rows)
    keys = sum(w.m_sizes) * d * (2 if folded else 1)
    uniq = 0
    for b in range(w.B):
        lo, hi = int(w.row_offsets[b]), int(w.row_offsets[b + 1])
        sel = set()
        for n in range(lo, hi):
            sel.update(int(x) for x in indices[n, :int(counts[n])])
        uniq += len(sel)
    row_w = 2 * H if projected else d
    values = uniq * row_w
    rows_io = 2 * N * d
    nbytes = es * (weights + keys + values + rows_io) + N * 4 + N * w.k_max * 4
    flops = 0 if folded else 2 * N * d * d                      # query
    rows = [int(w.row_offsets[b + 1] - w.row_offsets[b]) for b in range(w.B)]
    flops += sum(2 * rows[b] * int(w.m_sizes[b]) * d for b in range(w.B))
    flops += 2 * int(counts.sum()) * row_w                      # readout (projected or not)
    flops += 2 * N * (fuse1 + H * d + H)                        # fusion
    return float(nbytes), float(flops), int(uniq)


def kernel_bytes(name: str, w: workloads.Workload, uniq_values: int, projected: bool,
                 dense: bool = False) -> float:
    """HBM bytes one launch of a kernel must move (reads + writes).  `dense`:
    the step runs the dense-weights path (the selection writes the weights
    alpha as a bf16 hi / lo pair [N, P], P the longest memory rounded up to
    64, and the activation GEMM reads them with the transposed projected
    values [B, 2H, P])."""
    d, H, N = w.d, w.params["b_f1"].shape[0], w.N
    P = (max(int(m) for m in w.m_sizes) + 63) // 64 * 64
    es = 2 if w.dtype == "bf16" else 4
    scores = sum(int(w.row_offsets[b + 1] - w.row_offsets[b]) * int(w.m_sizes[b]) for b in range(w.B)) * 4
    if name == "query_proj":
        if projected:     # W_Q and the h-half of [W_f1 ; W_g1]; x, h in; q_hi, q_lo, G_h out
            return es * (d * d + 2 * H * d + 2 * N * d + 2 * N * d) + 4 * N * 2 * H
        return es * (d * d + N * d + 2 * N * d)
    if name == "fusion_h":        # the h-half of [W_f1 ; W_g1]; h in; G_h out
        return es * (2 * H * d + N * d) + 4 * N * 2 * H
    if name == "score_fusion_h":  # folded keys (hi, lo), the h-half of [W_f1 ; W_g1], x_h and h in; scores, G_h out
        return (2 * sum(w.m_sizes) * d + 2 * H * d + 2 * N * d) * es + scores + 4 * N * 2 * H
    if name == "score_folded":    # folded keys (hi, lo), x_h in; scores out
        return 2 * sum(w.m_sizes) * d * es + N * d * es + scores
    if name == "fuse_hidden":
        return es * (2 * H * 2 * d + 2 * N * d + N * 2 * H + 2 * H)
    if name == "fuse_out":
        return es * (d * H + N * H + d) + 4 * N * d
    if name == "score":
        keys = sum(w.m_sizes) * d * es
        return keys + 2 * N * d * es + scores
    if name == "readout":
        return uniq_values * d * es + N * d * (4 + es)
    if name == "select_fuse":     # scores in; projected rows, G_h, biases in; activations out
        return scores + uniq_values * 2 * H * es + 4 * N * 2 * H + es * (2 * H + N * 2 * H) + N * 4 + N * w.k_max * 4
    if name == "select_readout":
        return scores + uniq_values * d * es + N * d * (4 + es) + N * 4 + N * w.k_max * 4
    if name == "select":
        return scores + 3 * N * w.k_max * 4 + (N * P * 2 * es if dense else 0)
    if name == "act_gemm":        # alpha (hi, lo), transposed projected values, G_h, biases in; activations out
        return es * (2 * N * P + w.B * 2 * H * P + 2 * H + N * 2 * H) + 4 * N * 2 * H
    if name == "ln_query":
        return es * (2 * N * d + 4 * d)
    if name == "finalize":
        return es * (2 * N * d + N * H + 2 * d) + 4 * N * d
    return 0.0


# ---------------------------------------------------------------------------
# Clocks sampled during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.dev}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.2)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for nm, val in zip(names, parts[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(nm)
        os.unlink(self.path)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": float(max(mx)) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# Reference arm: the CPU oracle
# ---------------------------------------------------------------------------

def oracle_inputs(w: workloads.Workload):
    """The stored (bf16 / fp32) inputs as float64, exactly as the GPU sees them."""
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32

    def f64(a):
        return torch.from_numpy(np.ascontiguousarray(a)).to(dt).to(torch.float64).numpy()
    p = {k: f64(v) for k, v in w.params.items()}
    return p, f64(w.v), f64(w.h)


def time_oracle(w: workloads.Workload, min_seconds: float, max_rows: int = None,
                rows_per_call: int = None):
    """Run the oracle's retrieve+fuse on rows of the workload until
    min_seconds elapsed; returns (rows/s, rows, seconds, build seconds)."""
    import oracle
    p, v, h = oracle_inputs(w)
    mirror = w.dtype == "bf16"
    t0 = time.perf_counter()
    mem = oracle.build_memory(p, v, w.mask, mirror=mirror, ln_eps=float(np.float32(1e-5)))
    build_s = time.perf_counter() - t0
    rows_per_call = rows_per_call or w.N
    done, t_start, i = 0, time.perf_counter(), 0
    while True:
        sel = [(i * rows_per_call + j) % w.N for j in range(rows_per_call)]
        oracle.retrieve_fuse(p, mem, h, w.depth, w.row_offsets, w.row_scale, w.rho, w.k_min,
                             w.k_max, mirror=mirror, rows=sel, ln_eps=float(np.float32(1e-5)),
                             rms_eps=float(np.float32(1e-6)))
        done += rows_per_call
        i += 1
        el = time.perf_counter() - t_start
        if el >= min_seconds or (max_rows is not None and done >= max_rows):
            return done / el, done, el, build_s


def cores_used() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def max_over_ranks(value: float, dist, device) -> float:
    """The largest `value` over the ranks of the job (a replica job's step time
    is its slowest replica's); `dist` is torch.distributed or None (one rank)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def run_reference(args, w):
    """The reference arm: the CPU oracle as it stands, timed on this host's
    cores on the GPU arm's workload.  A step is an oracle retrieve+fuse over
    the workload's draft states (the memory is built once, untimed); when
    --steps such steps would take more than about two minutes, each step
    covers an evenly strided sample of the rows instead, and the line says so."""
    import oracle
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    p, v, h = oracle_inputs(w)
    mirror = w.dtype == "bf16"
    mem = oracle.build_memory(p, v, w.mask, mirror=mirror, ln_eps=float(np.float32(1e-5)))
    eps = dict(ln_eps=float(np.float32(1e-5)), rms_eps=float(np.float32(1e-6)))

    def one(rows):
        oracle.retrieve_fuse(p, mem, h, w.depth, w.row_offsets, w.row_scale, w.rho, w.k_min,
                             w.k_max, mirror=mirror, rows=rows, **eps)
    t0 = time.perf_counter()
    one(None)                                   # first warm-up step: all rows, to size the sample
    t_full = time.perf_counter() - t0
    rows_per_step = w.N
    budget_s = 120.0
    if t_full * args.steps > budget_s:
        rows_per_step = max(1, int(w.N * budget_s / (t_full * args.steps)))
    stride = max(1, w.N // rows_per_step)

    def rows_of(i):
        if rows_per_step >= w.N:
            return None
        return sorted({(i + j * stride) % w.N for j in range(rows_per_step)})
    for i in range(1, args.warmup):
        one(rows_of(i))
    t0 = time.perf_counter()
    for i in range(args.steps):
        one(rows_of(args.warmup + i))
    el = time.perf_counter() - t0
    value = rows_per_step * args.steps / el
    sample = (f"every step the whole {w.N}-row batch" if rows_per_step >= w.N else
              f"every step {rows_per_step} of the {w.N} rows (strided, rotating), the whole "
              f"batch taking {t_full:.2f} s")
    sample += "; memory built once (excluded)"
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": 1000 * el / args.steps, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "impl": "reference",
           "config": workload_config(w),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
                            "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))
    return 0


def workload_config(w: workloads.Workload) -> dict:
    return {"workload": w.name, "d_model": w.d, "memory_entries": [int(m) for m in w.m_sizes],
            "draft_states": w.N, "sequences": w.B, "rho": w.rho, "k_min": w.k_min,
            "k_max": w.k_max, "mlp_hidden": int(w.params["b_f1"].shape[0])}


# ---------------------------------------------------------------------------
# The GPU arm
# ---------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="fovea", choices=["fovea", "reference"])
    ap.add_argument("--workload", type=int, default=2)
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-supplemental", action="store_true")
    args = ap.parse_args()
    assert args.warmup >= 3, "at least 3 warm-up steps"

    spec = workloads.WORKLOADS[args.workload]
    w = workloads.generate(spec)
    if args.impl == "reference":
        return run_reference(args, w)

    from paper_2608_22883_gb300 import fovea

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    dev = torch.device("cuda", local)
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    weights = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dt).to(dev) for k, v in w.params.items()}
    params = fovea.Params(weights, d_model=w.d, mlp_hidden=w.params["b_f1"].shape[0],
                          max_depth=w.params["E_dep"].shape[0] - 1,
                          dtype=fovea.BF16 if w.dtype == "bf16" else fovea.FP32)
    v = torch.from_numpy(w.v).to(dt).to(dev)
    mask = torch.from_numpy(w.mask).to(dev) if w.mask is not None else None
    h_host = torch.from_numpy(w.h).to(dt).pin_memory()
    depth_host = torch.from_numpy(w.depth).pin_memory()
    h = h_host.to(dev)
    depth = depth_host.to(dev)
    row_scale = torch.from_numpy(w.row_scale).to(dev) if w.row_scale is not None else None

    # the memory build (once per image batch), timed with its per-kernel events
    # on a second build: the first loads the kernels' modules and is discarded
    torch.cuda.synchronize()
    fovea.build_memory(params, v, mask).destroy()
    torch.cuda.synchronize()
    fovea.timing_enable(True)
    t0 = time.perf_counter()
    mem = fovea.build_memory(params, v, mask)
    torch.cuda.synchronize()
    build_ms = 1000 * (time.perf_counter() - t0)
    build_kernels = {k: {"ms": t, "launches": n} for k, (t, n) in fovea.timing_read().items()}
    # the key / value projection GEMM: 2 * entries * (2 d) * d flops
    proj_ms = build_kernels.get("memory_proj", {}).get("ms")
    build_proj_tflops = (2.0 * sum(mem.valid_counts) * 2 * w.d * w.d / (proj_ms * 1e-3) / 1e12
                         if proj_ms else None)
    fovea.timing_enable(False)

    N, d, K = w.N, w.d, w.k_max
    ws = fovea.new_workspace(params, mem, w.row_offsets, K)
    # The step's inputs (h, depth) and outputs (h_hat, counts, indices) each
    # live in one contiguous buffer, so the end-to-end step moves them with
    # one host-to-device and one device-to-host copy.
    def packed(parts, device, pin=False):
        sizes = [int(np.prod(shp)) * torch.empty((), dtype=dt_).element_size() for shp, dt_ in parts]
        offs = np.cumsum([0] + [(b + 255) // 256 * 256 for b in sizes])
        buf = torch.empty(int(offs[-1]), dtype=torch.uint8, device=device)
        if pin:
            buf = buf.pin_memory()
        views = [buf[int(o):int(o) + b].view(dt_).view(shp) for o, b, (shp, dt_) in zip(offs, sizes, parts)]
        return buf, views
    out_parts = [((N, d), h.dtype), ((N,), torch.int32), ((N, K), torch.int32)]
    out_dev, (h_out, counts, indices) = packed(out_parts, dev)
    offs_c = fovea._offsets(w.row_offsets)
    flush_w = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flush_r = torch.ones(L2_FLUSH_BYTES // 8, dtype=torch.float32, device=dev)
    in_parts = [((N, d), h.dtype), ((N,), torch.int32)]
    in_dev, (h_in, depth_in) = packed(in_parts, dev)         # the step reads its inputs here
    in_host, (h_in_host, depth_in_host) = packed(in_parts, "cpu", pin=True)
    h_in_host.copy_(h_host)
    depth_in_host.copy_(depth_host)
    h_in.copy_(h)
    depth_in.copy_(depth)
    out_host, (h_out_host, counts_host, idx_host) = packed(out_parts, "cpu", pin=True)

    def step():
        fovea.retrieve_fuse(params, mem, h_in, depth_in, w.row_offsets, row_scale, w.rho, w.k_min,
                            K, h_out, ws, counts=counts, indices=indices, offsets_c=offs_c)

    def flush(i):
        # evict everything: write 512 MB, then read 256 MB so the lines L2 holds
        # when the step starts are clean (no write-back charged to the step)
        flush_w.fill_(i & 0xFF)
        flush_r.sum()

    stream = torch.cuda.current_stream()
    # The step is timed in two forms: one CUDA-graph replay per step (the
    # form a decoding loop captures), and the plain API call (its kernels
    # enqueued by fovea_retrieve_fuse itself, the host work overlapping the
    # L2 flush before it).  The headline takes the plain call.
    cap = torch.cuda.Stream()
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        for _ in range(3):
            step()
    stream.wait_stream(cap)
    torch.cuda.synchronize()
    g_plain = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_plain, stream=cap):
        step()
    # end to end as a graph: the host inputs copied in, the step, the results
    # copied back (pinned host buffers)
    g_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_e2e, stream=cap):
        in_dev.copy_(in_host, non_blocking=True)
        step()
        out_host.copy_(out_dev, non_blocking=True)
    torch.cuda.synchronize()

    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)

    def timed(run, n, seed):
        ts = []
        for i in range(n):
            flush(seed + i)
            e0.record(stream)
            run()
            e1.record(stream)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1))
        return ts

    timed(step, args.warmup, 0)
    timed(g_plain.replay, args.warmup, 0)
    fovea.sync_errors(ws)

    # ---- timed region: K steps (plain API calls), L2 flushed before each ----
    clocks = ClockSampler(local)
    clocks.start()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    step_ms = timed(step, args.steps, 7)
    torch.cuda.synchronize()
    wall_s = time.perf_counter() - t_wall
    graph_ms_l = timed(g_plain.replay, min(args.steps, 500), 11)
    # warm, back to back (labelled as such; not the headline): the same API
    # call repeated without an L2 flush, one event pair around the run
    n_warm = min(args.steps, 200)
    torch.cuda.synchronize()
    e0.record(stream)
    for i in range(n_warm):
        step()
    e1.record(stream)
    e1.synchronize()
    warm_ms = e0.elapsed_time(e1) / n_warm
    if dist is not None:
        dist.barrier()
    clk = clocks.stop()
    ms = float(np.mean(step_ms))
    fovea.sync_errors(ws)
    ms = max_over_ranks(ms, dist, dev)
    graph_ms = max_over_ranks(float(np.mean(graph_ms_l)), dist, dev)
    value = world * N / (ms / 1000.0)

    # ---- kernel-timing pass: the same step with an event pair around every
    # kernel (event nodes add a gap at each kernel boundary, so these per-kernel
    # durations are upper bounds) ----
    n_kt = min(args.steps, 500)
    per_kernel = {}
    kt_ms = []
    fovea.timing_enable(True)            # per-kernel event nodes in the timed graph; kept
    g_timed = torch.cuda.CUDAGraph()     # enabled while the graph is replayed
    with torch.cuda.graph(g_timed, stream=cap):
        step()
    torch.cuda.synchronize()
    for i in range(n_kt):
        flush(i)
        e0.record(stream)
        g_timed.replay()
        e1.record(stream)
        e1.synchronize()
        kt_ms.append(e0.elapsed_time(e1))
        for name, (tot, n) in fovea.timing_read().items():
            a = per_kernel.setdefault(name, [0.0, 0])
            a[0] += tot
            a[1] += n
    ms_hooks = float(np.mean(kt_ms))

    # ---- end to end: host buffers in, the step, results back to host (one
    # graph: the copies are memcpy nodes around the step's kernels) ----
    fovea.timing_enable(False)
    e2e_ms_l = timed(g_e2e.replay, n_kt, 3)
    e2e_ms = max_over_ranks(float(np.mean(e2e_ms_l)), dist, dev)
    h2d = in_host.numel()
    d2h = out_host.numel()
    assert torch.equal(h_out_host, h_out.cpu())
    # ---- the public API call end to end on the host clock: copy the inputs
    # in, call fovea_retrieve_fuse (argument checks, planning, launches),
    # copy the outputs back, synchronise; no graph, no L2 flush ----
    wall_l = []
    for i in range(min(args.steps, 300) + 3):
        t0 = time.perf_counter()
        in_dev.copy_(in_host, non_blocking=True)
        step()
        out_host.copy_(out_dev, non_blocking=True)
        stream.synchronize()
        if i >= 3:
            wall_l.append(time.perf_counter() - t0)
    api_wall_ms = 1000 * float(np.median(wall_l))
    api_host_l = []
    for i in range(200):             # host time of the call alone (the GPU catches up after)
        t0 = time.perf_counter()
        step()
        api_host_l.append(time.perf_counter() - t0)
        if i % 16 == 15:
            stream.synchronize()
    stream.synchronize()
    api_host_us = 1e6 * float(np.median(api_host_l))

    # ---- roofline ----
    c_np, i_np = counts.cpu().numpy(), indices.cpu().numpy()
    dense = "act_gemm" in per_kernel
    projected = "select_fuse" in per_kernel or dense
    folded = "score_folded" in per_kernel or "score_fusion_h" in per_kernel
    # the method's algorithmic bytes (full fusion weights, value rows), and
    # what this path's step moves (projected values: the h-half weights and
    # 2H-wide memory rows; folded keys: no W_Q, hi / lo keys)
    nbytes, flops, uniq = step_cost(w, c_np, i_np, False)
    nbytes_path, flops_path, _ = step_cost(w, c_np, i_np, projected, folded)
    peaks, peak_src = load_peaks()
    t_hbm = nbytes / (peaks["hbm_gbs"] * 1e9)
    t_tc = flops / (peaks["bf16_tflops"] * 1e12)
    t_roof = max(t_hbm, t_tc)
    t_roof_path = max(nbytes_path / (peaks["hbm_gbs"] * 1e9), flops_path / (peaks["bf16_tflops"] * 1e12))
    kern = {name: {"ms_avg": tot / max(n, 1), "launches": n} for name, (tot, n) in per_kernel.items()}
    dom = max(kern, key=lambda k: kern[k]["ms_avg"] * kern[k]["launches"])
    dom_bytes = kernel_bytes(dom, w, uniq, projected, dense)
    achieved = dom_bytes / (kern[dom]["ms_avg"] / 1000.0) / 1e9
    launches_per_step = sum(k["launches"] for k in kern.values()) / max(n_kt, 1)
    launches = int(round(launches_per_step * args.steps))
    total_kernel_ms = sum(k["ms_avg"] * k["launches"] for k in kern.values())
    traffic = None
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tpath):
        try:
            with open(tpath) as f:
                tr = json.load(f)
            ent = tr.get(w.name, {}).get(dom)
            if ent and ent.get("kernel_sha") == _kernel_sha(ent.get("files")):
                traffic = ent["bytes_per_launch"]
        except Exception:
            traffic = None

    cfg = workload_config(w)
    cfg.update({"l2": "flushed before every step outside the per-step events (512 MB write, then a 256 MB read so the evicted lines are clean)",
                "launch": f"one fovea_retrieve_fuse call per step ({len(kern)} kernels, programmatic "
                          "dependent launch between them)",
                "parallelism": f"replicas x{world}"})
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
        "config": cfg,
        "roofline": {"kernel": dom, "bound": "hbm", "achieved": achieved,
                     "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                     "traffic": traffic, "algorithmic_bytes": dom_bytes,
                     "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
                     else "fallback 6.8 TB/s"},
        "step_roofline": {"bytes": nbytes, "flops": flops, "unique_value_rows": uniq,
                          "t_roof_us": 1e6 * t_roof, "bound": "hbm" if t_hbm >= t_tc else "tensor",
                          "frac": t_roof / (ms / 1000.0),
                          "this_path": {"bytes": nbytes_path, "flops": flops_path,
                                        "t_roof_us": 1e6 * t_roof_path,
                                        "frac": t_roof_path / (ms / 1000.0),
                                        "projected_values": projected,
                                        "folded_keys": folded},
                          "peaks": f"{peak_src}: {peaks['hbm_gbs']} GB/s, {peaks['bf16_tflops']} TF/s"},
        "kernels": {k: {"us_avg": 1000 * v["ms_avg"], "launches": v["launches"],
                        "algorithmic_bytes": kernel_bytes(k, w, uniq, projected, dense),
                        "gbs": kernel_bytes(k, w, uniq, projected, dense) / (v["ms_avg"] / 1000.0) / 1e9}
                    for k, v in kern.items()},
        "ms_per_step_graph_replay": graph_ms,
        "ms_per_step_kernel_timing_pass": ms_hooks,
        "kernel_ms_per_step": total_kernel_ms / max(n_kt, 1),
        "gpu_launches": launches,
        "ms_per_step_warm_back_to_back": warm_ms,
        "memory_build_ms": build_ms,
        "memory_build_kernels": build_kernels,
        "memory_build_proj_tflops": build_proj_tflops,
        "clocks": clk,
        "e2e": {"value": world * N / (e2e_ms / 1000.0), "unit": UNIT, "ms_per_step": e2e_ms,
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                "form": "one CUDA graph per step: input copy from pinned host memory, the step, "
                        "output copy back; CUDA events on the launching stream"},
        "api_call_host_clock": {"value": world * N / (api_wall_ms / 1000.0), "unit": UNIT,
                                "ms_per_step": api_wall_ms, "host_us_per_call": api_host_us,
                                "form": "per step on the host clock: input copy in, "
                                        "fovea_retrieve_fuse through the Python binding, output "
                                        "copy back, stream synchronise (median)"},
        "wall_s_timed_region": wall_s,
    }
    # supplemental points (not the headline): small N and the paper's other
    # retrieval settings, cold L2, one plain call per step
    if not args.no_supplemental:
        out["supplemental"] = supplemental(fovea, params, mem, w, h_in, depth_in, row_scale, flush,
                                           min(args.steps, 300))
        if w.dtype == "bf16" and w.B == 1:
            out["supplemental"]["lm_head_topk_v32000_k6"] = lm_head_point(
                fovea, h_out, flush, min(args.steps, 300), peaks, step=step)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate, rows, secs, build_s = time_oracle(w, args.cpu_seconds)
        out["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
                               "sample": f"{rows} draft states ({rows // w.N} oracle steps of the "
                                         f"{w.N}-row batch) in {secs:.1f} s; memory build "
                                         f"({build_s:.1f} s) excluded"}
    if rank == 0:
        print(json.dumps(out))
    if dist is not None:
        dist.destroy_process_group()
    return 0


def _time_calls(call, flush, n_steps, warm=3):
    """Mean CUDA-event time (ms) of `call` on the current stream, L2 flushed
    before each, after `warm` untimed calls."""
    stream = torch.cuda.current_stream()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    for i in range(warm):
        flush(i)
        call()
    ts = []
    for i in range(n_steps):
        flush(i)
        e0.record(stream)
        call()
        e1.record(stream)
        e1.synchronize()
        ts.append(e0.elapsed_time(e1))
    return float(np.mean(ts))


def supplemental(fovea, params, mem, w, h, depth, row_scale, flush, n_steps):
    """Per-step latency of the small-N regime (the root and its K_c = 6
    depth-1 children of one sequence), of the depth gate at the paper's
    l <= 1, and of the paper's other retrieval settings, on the same memory
    and hidden states.  Each is timed like the headline: CUDA events on the
    launching stream around one plain call, L2 flushed before it."""
    cases = []
    if w.B == 1 and w.N >= 7:
        cases.append(("small_n_7", 7, w.rho, w.k_min, w.k_max, None))
    cases.append(("depth_gate_l1", w.N, w.rho, w.k_min, w.k_max, 1))
    cases.append(("paper_defaults_rho0.8_kmin32_kmax256", w.N, 0.8, 32, 256, None))
    cases.append(("fixed_top16", w.N, w.rho, 16, 16, None))
    m_max = int(max(w.m_sizes))
    if m_max <= 1024:
        cases.append((f"dense_k{m_max}", w.N, 1.0, m_max, m_max, None))
    fovea.timing_enable(False)
    out = {}
    for name, n, rho, kmin, kmax, l_max in cases:
        offs = list(w.row_offsets) if n == w.N else [0, n]
        hn, dn = h[:n].contiguous(), depth[:n].contiguous()
        rs = row_scale[:n].contiguous() if row_scale is not None else None
        ws = fovea.new_workspace(params, mem, offs, kmax)
        h_out = torch.empty_like(hn)
        counts = torch.empty(n, dtype=torch.int32, device=hn.device)
        offs_c = fovea._offsets(offs)

        def step():
            fovea.retrieve_fuse(params, mem, hn, dn, offs, rs, rho, kmin, kmax, h_out, ws,
                                counts=counts, offsets_c=offs_c, l_max=l_max)
        ms = _time_calls(step, flush, n_steps)
        fovea.sync_errors(ws)
        c = counts.cpu().numpy()
        out[name] = {"draft_states": n, "rho": rho, "k_min": kmin, "k_max": kmax,
                     "l_max": l_max, "us_per_step": 1000 * ms, "value": n / (ms / 1000.0),
                     "unit": UNIT, "mean_count": float(c.mean()), "steps": n_steps}
    return out


def lm_head_point(fovea, h_hat, flush, n_steps, peaks, vocab=32000, k_c=6, seed=7, step=None):
    """The draft logits and K_c candidates (fovea_lm_head_topk) on the step's
    own h_hat: a synthetic bf16 W_LM [vocab, d] ~ N(0, 1/d), drawn on the
    device from a seeded generator; one plain call per step, L2 flushed
    before each, CUDA events on the launching stream.  With `step` (the
    draft step writing h_hat), also the step followed by the LM head on the
    same stream in one timed region: the LM head's weight stream starts while
    the step's last kernel runs (programmatic dependent launch)."""
    N, d = h_hat.shape
    gen = torch.Generator(device=h_hat.device)
    gen.manual_seed(seed)
    W = (torch.randn((vocab, d), generator=gen, device=h_hat.device) / math.sqrt(d)).to(torch.bfloat16)
    ws = fovea.lm_head_workspace(vocab, d, N, k_c)
    logits = torch.empty((N, vocab), dtype=torch.float32, device=h_hat.device)
    ms = _time_calls(lambda: fovea.lm_head_topk(W, h_hat, k_c, ws, logits=logits), flush, n_steps)
    ms_c = _time_calls(lambda: fovea.lm_head_topk(W, h_hat, k_c, ws, write_logits=False), flush, n_steps)
    after = None
    if step is not None:
        def step_then_head():
            step()
            fovea.lm_head_topk(W, h_hat, k_c, ws, logits=logits)
        ms_s = _time_calls(step, flush, n_steps)
        ms_sh = _time_calls(step_then_head, flush, n_steps)
        after = {"us_step": 1000 * ms_s, "us_step_then_lm_head": 1000 * ms_sh,
                 "us_lm_head_after_step": 1000 * (ms_sh - ms_s)}
    fovea.sync_errors(ws)
    # algorithmic bytes: W_LM once, h_hat in, the logits out (first form
    # only), the per-tile candidates out and back in for the merge, the
    # K_c candidates (index, value) out
    tiles = (vocab + 255) // 256
    base = vocab * d * 2 + N * d * 2 + 2 * N * tiles * k_c * 8 + N * k_c * 8
    nbytes = base + N * vocab * 4
    gbs = nbytes / (ms / 1000.0) / 1e9
    del W, logits
    return {"vocab": vocab, "d_model": d, "draft_states": N, "k_c": k_c, "us_per_call": 1000 * ms,
            "algorithmic_bytes": nbytes, "achieved_gbs": gbs, "frac_of_measured_hbm": gbs / peaks["hbm_gbs"],
            "after_step": after,
            "candidates_only": {"us_per_call": 1000 * ms_c, "algorithmic_bytes": base,
                                "frac_of_measured_hbm": base / (ms_c / 1000.0) / 1e9 / peaks["hbm_gbs"]},
            "steps": n_steps, "w_lm": "synthetic N(0, 1/d), bf16"}


def _kernel_sha(files=None) -> str:
    """Hash of the sources a kernel is built and launched from (paths relative
    to the repository root; default: every file of csrc/)."""
    import hashlib
    hsh = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_22883_gb300", "csrc")
    paths = ([os.path.join(ROOT, f) for f in files] if files
             else [os.path.join(csrc, f) for f in sorted(os.listdir(csrc))])
    for path in paths:
        with open(path, "rb") as fh:
            hsh.update(fh.read())
    return hsh.hexdigest()[:16]


if __name__ == "__main__":
    sys.exit(main())
