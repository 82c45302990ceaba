#!/usr/bin/env python3
"""Benchmark: chunked causal prefill attention (MOCAP's hot path) on GB300.

One step = one pass of the whole hot path over one prompt: LBCP boundaries
(host), then for every chunk the KV append and the chunk attention.  The
default workload is the 131072-token Llama-3-70B attention shape (64 q-heads,
8 kv-heads, d=128) in 32 LBCP chunks.  Inputs are larger than L2 (Q 2 GiB,
K/V 256 MiB each), so no flush is needed between steps.

Prints ONE JSON line (rank 0).  ``--impl reference`` times the float64 CPU
oracle instead, on a bounded row sample of the same workload.

Under torchrun each rank runs an independent replica on its own GPU (the
path has no exchange step); value = all ranks' work / the slowest rank.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "chunk-attn TFLOP/s & % GB300 BF16 tensor peak; prefill tokens/s"
FALLBACK_PEAK_TFLOPS = 1700.0  # sustained bf16, used only without MEASURED_PEAKS.json
FALLBACK_BURST_TFLOPS = 1900.0  # burst bf16, likewise
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", type=int, default=4)
    ap.add_argument("--append-mode", choices=["serial", "fused", "overlap"], default="overlap",
                    help="how chunk K/V reach the cache in the timed steps "
                         "(ChunkedPrefill append_mode)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-graph", action="store_true",
                    help="skip the CUDA-graph replay measurement")
    ap.add_argument("--no-projection", action="store_true",
                    help="skip the QKV projection + RoPE + append measurement")
    ap.add_argument("--hidden", type=int, default=8192,
                    help="hidden size for the projection measurement (Llama-3-70B: 8192)")
    ap.add_argument("--no-append-modes", action="store_true",
                    help="skip the append measurements after the timed region (the append "
                         "graphs and the comparison of the three append modes)")
    ap.add_argument("--no-last-row", action="store_true",
                    help="skip the last-row-only attention measurement")
    ap.add_argument("--no-uniform", action="store_true",
                    help="skip the uniform-boundary per-chunk latency comparison")
    ap.add_argument("--cpu-rows-per-chunk", type=int, default=4)
    ap.add_argument("--case", default=None,
                    help="profiling case 'prefix,len,Hq,Hkv,d': one chunk attention launch "
                         "repeated warmup+steps times (no JSON metric line)")
    ap.add_argument("--case-split", choices=["none", "auto"], default="none",
                    help="with --case: 'auto' passes the library's split-KV workspace, as "
                         "the prompt pipeline does (the launch may split and add a combine)")
    ap.add_argument("--case-host-copy", default=None,
                    help="profiling case 'bytes,up|down,0|1': one host <-> device copy by the "
                         "SMs (mocap_copy_from_host / _to_host), repeated (no JSON line)")
    ap.add_argument("--case-append", default=None,
                    help="profiling case 'rows,Hkv,d': one KV append launch repeated "
                         "warmup+steps times")
    ap.add_argument("--case-append-overlap", action="store_true",
                    help="with --case-append: time mocap_kv_append_overlap (the one-warp "
                         "kernel meant to run beside attention) instead of mocap_kv_append")
    ap.add_argument("--case-qkv", default=None,
                    help="profiling case 'len,hidden,Hq,Hkv,d': one QKV projection launch "
                         "repeated warmup+steps times")
    ap.add_argument("--case-last-row", default=None,
                    help="profiling case 'keys,Hq,Hkv,d': one last-row attention launch "
                         "repeated warmup+steps times")
    return ap.parse_args()


# ------------------------------------------------------------------ helpers --
def attn_flops(bounds_list, n_q_heads, head_dim):
    """Algorithmic FLOP: 4 * Hq * d per causal (query, key) pair; pairs per
    chunk c_i * p_i + c_i (c_i + 1) / 2 (exact, no masked-tile waste)."""
    per_chunk = []
    for bounds in bounds_list:
        per_chunk.append([4 * n_q_heads * head_dim *
                          ((b1 - b0) * b0 + (b1 - b0) * (b1 - b0 + 1) // 2)
                          for b0, b1 in zip(bounds[:-1], bounds[1:])])
    return per_chunk


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"bf16_tflops_sustained": FALLBACK_PEAK_TFLOPS, "hbm_gbs": FALLBACK_HBM_GBS}, \
            "fallback"


def kernel_source_hash():
    """Hash of the attention kernel's device source (the kernel header and the
    PTX wrappers it uses), which the committed DRAM captures were taken on."""
    h = hashlib.sha256()
    for f in ("attn_kernel.cuh", "sm103_ptx.cuh"):
        with open(os.path.join(ROOT, "paper_2606_22968_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def attn_min_bytes(prefix, length, n_q_heads, n_kv_heads, head_dim):
    """Algorithmic HBM bytes of one chunk attention launch: K and V of the
    prefix plus the chunk read once, Q read, O written (bf16), LSE written
    (fp32)."""
    kv = 2 * (prefix + length) * n_kv_heads * head_dim * 2
    return kv + 2 * length * n_q_heads * head_dim * 2 + 4 * length * n_q_heads


def read_traffic_cases():
    """Single-kernel ncu captures of chunk_attn_kernel (one launch each) from
    the committed summary: {(prefix, len, Hq, Hkv, d): DRAM bytes}, or None
    when the summary was not taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", "chunk_attn_dram_traffic.txt")
    try:
        cases, src = {}, None
        with open(path) as f:
            for line in f:
                line = line.strip()
                if not line or line.startswith("#"):
                    continue
                key, val = line.split(":", 1)
                if key == "kernel_source_sha256_16":
                    src = val.strip()
                elif key == "case":
                    fields = val.split()
                    shape = tuple(int(x) for x in fields[:5])
                    kv = dict(x.split("=") for x in fields[5:])
                    cases[shape] = float(kv["dram_bytes"])
        if src != kernel_source_hash() or not cases:
            return None
        return cases
    except Exception:
        return None


def ncu_traffic(bounds, n_q_heads, n_kv_heads, head_dim):
    """DRAM bytes per attention launch of a single-request prompt, averaged
    over its chunks.  Each chunk's bytes are its algorithmic minimum times the
    measured ratio (DRAM bytes / minimum) of the captured shapes, linearly
    interpolated in the chunk's key count prefix + len (captured shapes of
    the same heads and head dimension; outside their range the nearest
    ratio).  None without current captures of these heads."""
    cases = read_traffic_cases()
    if cases is None:
        return None
    pts = sorted((p + n, b / attn_min_bytes(p, n, hq, hkv, d))
                 for (p, n, hq, hkv, d), b in cases.items()
                 if (hq, hkv, d) == (n_q_heads, n_kv_heads, head_dim))
    if not pts:
        return None

    def ratio(keys):
        if keys <= pts[0][0]:
            return pts[0][1]
        for (x0, r0), (x1, r1) in zip(pts, pts[1:]):
            if keys <= x1:
                return r0 + (r1 - r0) * (keys - x0) / (x1 - x0)
        return pts[-1][1]

    alg = [attn_min_bytes(b0, b1 - b0, n_q_heads, n_kv_heads, head_dim)
           for b0, b1 in zip(bounds[:-1], bounds[1:])]
    est = [a * ratio(b1) for a, b1 in zip(alg, bounds[1:])]
    return {"traffic": sum(est) / len(est), "algorithmic": sum(alg) / len(alg),
            "captured_shapes": len(pts)}


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            import tempfile
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.close()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax = float(parts[2])
                except ValueError:
                    continue
                for name, val in zip(names, parts[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------- CPU oracle --
def oracle_sample_plan(bounds, rows_per_chunk, step_index):
    """(chunk, rows) items the oracle evaluates in one sampled step: for every
    chunk, the last row plus evenly spread rows shifted by the step index;
    chunks are visited last-first, then first, then alternating inwards so a
    time-bounded prefix of the plan still spans short and long prefixes."""
    n_chunks = len(bounds) - 1
    order, lo, hi = [], 0, n_chunks - 1
    while lo <= hi:
        order.append(hi)
        if lo != hi:
            order.append(lo)
        lo, hi = lo + 1, hi - 1
    plan = []
    for i in order:
        n = bounds[i + 1] - bounds[i]
        rows = {n - 1}
        for r in range(1, rows_per_chunk):
            rows.add((r * n // rows_per_chunk + 37 * step_index) % n)
        plan.append((i, sorted(rows)))
    return plan


def _oracle_worker(args):
    """Runs in a spawned process: times the oracle over sampled rows, each
    step stopping after `budget_s` seconds (at least one item)."""
    (q_items, k_bits, v_bits, bounds, plans, scale, budget_s, threads) = args
    import numpy as np
    from oracle import attention as A
    k = A.bf16_bits_to_f64(k_bits)
    v = A.bf16_bits_to_f64(v_bits)
    times, flops, done = [], [], []
    for plan, qs in zip(plans, q_items):
        t0 = time.perf_counter()
        fl, n_done = 0, 0
        for (i, rows), q_bits in zip(plan, qs):
            b0, b1 = bounds[i], bounds[i + 1]
            r = np.array(rows)
            q_rows = A.bf16_bits_to_f64(q_bits)
            q_full = np.zeros((int(r.max()) + 1,) + q_rows.shape[1:])
            q_full[r] = q_rows
            A.chunk_attention(q_full, k[:b1], v[:b1], b0, scale, rows=r)
            fl += sum(4 * q_rows.shape[1] * q_rows.shape[2] * (b0 + x + 1) for x in rows)
            n_done += 1
            if time.perf_counter() - t0 > budget_s:
                break
        times.append(time.perf_counter() - t0)
        flops.append(fl)
        done.append(n_done)
    return times, flops, done


def run_oracle_sample(q, k, v, bounds, scale, n_steps, rows_per_chunk, budget_s):
    """Time the oracle on sampled rows (q/k/v: torch tensors on any device)."""
    import multiprocessing as mp
    import torch
    threads = os.cpu_count() or 1
    plans = [oracle_sample_plan(bounds, rows_per_chunk, s) for s in range(n_steps)]
    q_items = []
    for plan in plans:
        items = []
        for i, rows in plan:
            idx = torch.as_tensor([bounds[i] + x for x in rows], device=q.device)
            items.append(q[idx].cpu().view(torch.int16).numpy())
        q_items.append(items)
    k_bits = k.cpu().view(torch.int16).numpy()
    v_bits = v.cpu().view(torch.int16).numpy()
    env_keys = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS")
    saved = {x: os.environ.get(x) for x in env_keys}
    for x in env_keys:
        os.environ[x] = str(threads)  # inherited by the spawned worker
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(1) as pool:
            times, flops, done = pool.apply(
                _oracle_worker, ((q_items, k_bits, v_bits, bounds, plans, scale, budget_s,
                                  threads),))
    finally:
        for x, val in saved.items():
            if val is None:
                os.environ.pop(x, None)
            else:
                os.environ[x] = val
    return times, flops, done, threads


# --------------------------------------------------------------- main arms --
def init_dist(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world, device):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_rank, ms_per_step_max, world):
    """Whole-job rate of N independent replicas: every rank processed the same
    units per step; the slowest rank's step time bounds the job."""
    return world * units_per_rank / (ms_per_step_max * 1e-3)


def reference_arm(args, rank, world):
    """The float64 oracle, timed on the host cores on a bounded sample."""
    import torch
    from paper_2606_22968_gb300 import workloads
    from oracle import partition as P
    if rank != 0:
        return 0
    w = workloads.get(args.workload)
    bounds = P.boundaries(w.seq_lens[0], w.num_chunks[0], 128, w.mode)
    q, k, v = workloads.make_qkv(w, "cpu")
    n = args.steps + args.warmup
    budget = max(2.0, min(15.0, 150.0 / n))
    times, flops, done, threads = run_oracle_sample(q, k, v, bounds, w.scale, n,
                                                    args.cpu_rows_per_chunk, budget)
    t = sum(times[args.warmup:])
    fl = sum(flops[args.warmup:])
    value = fl / t / 1e12
    sample = (f"per step: up to {args.cpu_rows_per_chunk} rows x all {w.n_q_heads} heads of "
              f"each chunk, chunks visited last/first alternately until ~{budget:.0f} s "
              f"(chunks done per step: {done}); float64 oracle")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000 * t / max(1, args.steps), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {**w.describe(), "workload": w.name},
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def ours_arm(args, rank, world, local):
    import torch
    import paper_2606_22968_gb300 as m
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill

    m._lib.load()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workloads.get(args.workload)
    q, k, v = workloads.make_qkv(w, dev)
    # one compute stream in the timed region: chunk i's events then time its
    # launch alone (per-chunk latency, the roofline's per-launch duration);
    # consecutive chunks on two streams are measured after it
    pf = ChunkedPrefill(w, dev, append_mode=args.append_mode, chunk_streams=1)
    steps_plan = pf.steps()
    n_chunks = len(steps_plan)
    stream = torch.cuda.current_stream(dev)

    flops_chunks = attn_flops(pf.bounds, w.n_q_heads, w.head_dim)
    # chunks whose key range the library splits (each adds a combine launch)
    n_combines = 0
    if pf.single and pf.workspace is not None:
        b = pf.bounds[0]
        n_combines = sum(1 for i in range(len(b) - 1)
                         if m.mocap_chunk_attn_workspace_size(b[i], b[i + 1] - b[i], w.n_q_heads,
                                                              w.n_kv_heads, w.head_dim) > 0)
    # per step (chunk index k): attention FLOP of every (request, k)
    step_flops = [sum(flops_chunks[r][c] for r, c in st) for st in steps_plan]
    total_flops = sum(step_flops)
    row_bytes = w.n_kv_heads * w.head_dim * 2

    def rows_of(step):
        return sum(pf.bounds[r][c + 1] - pf.bounds[r][c] for r, c in step)

    append_bytes = 2 * 2 * w.total_tokens * row_bytes  # K, V x (read + write)
    # only step 0's chunks are appended on the compute stream before their
    # attention; the rest go to the cache beside the attention launches
    # (second stream, or inside the launch; ChunkedPrefill.append_mode)
    standalone_bytes = 2 * 2 * rows_of(steps_plan[0]) * row_bytes
    if pf.append_mode == "serial":
        standalone_bytes = append_bytes

    def one_step(ev=None):
        pf.partition()
        pf.run(q, k, v, stream, ev)

    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize(dev)
    if m.mocap_last_device_status() != m.MOCAP_OK:
        raise RuntimeError("device wait expired during warm-up")

    evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n_chunks)]
           for _ in range(args.steps)]
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize(dev)
    clocks.start()
    time.sleep(0.3)  # let the sampler start before load
    start.record(stream)
    for s in range(args.steps):
        one_step(evs[s])
    end.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop()
    status = m.mocap_last_device_status()
    if status != m.MOCAP_OK:
        raise RuntimeError(f"device status {m.mocap_status_string(status)}")

    ms_total = start.elapsed_time(end)
    ms_total = max_over_ranks(ms_total, world, dev)
    ms_step = ms_total / args.steps
    attn_ms = [[evs[s][c][1].elapsed_time(evs[s][c][2]) for c in range(n_chunks)]
               for s in range(args.steps)]
    app_ms = [[evs[s][c][0].elapsed_time(evs[s][c][1]) for c in range(n_chunks)]
              for s in range(args.steps)]
    attn_step_ms = [sum(x) for x in attn_ms]
    app_step_ms = [sum(x) for x in app_ms]
    per_chunk = [statistics.median(attn_ms[s][c] for s in range(args.steps))
                 for c in range(n_chunks)]
    cv = statistics.pstdev(per_chunk) / statistics.mean(per_chunk) if n_chunks > 1 else 0.0

    value = replica_throughput(total_flops, ms_step, world) / 1e12
    tokens_per_s = replica_throughput(w.total_tokens, ms_step, world)
    peaks, peak_src = load_peaks()
    # The denominator for a run held by the power cap is the sustained cuBLAS
    # figure (measured under the same cap, at a known clock); a run that
    # never reached the cap is compared with the burst figure.
    capped = "sw_power_cap" in (clk.get("reasons") or [])
    if capped:
        peak_name = "bf16_tflops_sustained"
        peak = float(peaks.get(peak_name, FALLBACK_PEAK_TFLOPS))
    else:
        peak_name = "bf16_tflops"
        peak = float(peaks.get(peak_name, FALLBACK_BURST_TFLOPS))
    attn_avg_ms = statistics.mean(attn_step_ms)
    achieved = total_flops / (attn_avg_ms * 1e-3) / 1e12
    traffic = ncu_traffic(pf.bounds[0], w.n_q_heads, w.n_kv_heads, w.head_dim) \
        if pf.single else None
    alg_bytes = statistics.mean(
        attn_min_bytes(b0, b1 - b0, w.n_q_heads, w.n_kv_heads, w.head_dim)
        for bnd in pf.bounds for b0, b1 in zip(bnd[:-1], bnd[1:]))
    # The sustained peak was measured at its own median SM clock; at the
    # bench's median clock the same tensor pipe delivers peak * f / f_peak.
    peak_mhz = (peaks.get("clocks_under_load") or {}).get("sm_mhz_median")
    frac_clock = None
    if capped and peak_mhz and clk.get("sm_mhz"):
        frac_clock = achieved / (peak * clk["sm_mhz"] / float(peak_mhz))
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    app_gbs = standalone_bytes / (statistics.mean(app_step_ms) * 1e-3) / 1e9

    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {**w.describe(), "workload": w.name,
                   "l2": "inputs larger than L2 (no flush): Q %.1f GiB, K+V %.2f GiB" % (
                       q.numel() * 2 / 2**30, 2 * k.numel() * 2 / 2**30),
                   "parallelism": "replicas" if world > 1 else "single-gpu"},
        "prefill_tokens_per_s": tokens_per_s,
        "attn_tflops_kernel_only": achieved,
        "attn_frac_of_peak": achieved / peak,
        "per_chunk_attn_ms": {"min": min(per_chunk), "max": max(per_chunk),
                              "max_over_min": max(per_chunk) / min(per_chunk), "cv": cv,
                              "ms": [round(t, 4) for t in per_chunk],
                              # each step's attention FLOP / its median launch time,
                              # and that rate's fraction of the sustained peak
                              "tflops": [round(f / (t * 1e-3) / 1e12, 1)
                                         for f, t in zip(step_flops, per_chunk)],
                              "frac_of_peak_min": min(f / (t * 1e-3) / 1e12 for f, t in
                                                      zip(step_flops, per_chunk)) / peak,
                              "frac_of_peak_max": max(f / (t * 1e-3) / 1e12 for f, t in
                                                      zip(step_flops, per_chunk)) / peak},
        "append": {"bytes_per_step": append_bytes,
                   "standalone_bytes_per_step": standalone_bytes,
                   "fused_bytes_per_step": append_bytes - standalone_bytes,
                   "gb_per_s": app_gbs, "frac_of_hbm": app_gbs / hbm,
                   "ms_per_step": statistics.mean(app_step_ms),
                   "note": "gb_per_s: the appends on the compute stream (step 0's chunks "
                           "unless append_mode is serial) between events in the timed steps; "
                           f"append_mode {pf.append_mode}"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak,
                     "peak_source": f"{peak_name} ({peak_src}; "
                                    f"{'power cap active' if capped else 'power cap not reached'}"
                                    " in the timed region)",
                     "frac_at_peak_clock": frac_clock,
                     "clock_note": (f"achieved / (peak x bench median SM clock {clk.get('sm_mhz')}"
                                    f" MHz / peak's median SM clock {peak_mhz} MHz)") if capped
                     else "the burst peak's clock is not recorded: no clock-scaled fraction",
                     "kernel": "chunk_attn_kernel",
                     "traffic": None if traffic is None else traffic["traffic"],
                     "algorithmic_bytes": alg_bytes,
                     "traffic_over_algorithmic": None if traffic is None else
                     traffic["traffic"] / traffic["algorithmic"],
                     "traffic_unit": "bytes per launch (avg over the step's launches)",
                     "traffic_source": None if traffic is None else
                     (f"single-launch ncu captures of {traffic['captured_shapes']} chunk shapes "
                      "(profiles/chunk_attn_dram_traffic.txt), DRAM/minimum ratio "
                      "interpolated in keys per chunk")},
        "clocks": clk,
        # our kernels per timed region: one append per (request, chunk) (in
        # fused mode only step 0's; the others ride in the attention
        # launches), one attention launch per step, one split-KV combine per
        # split chunk
        "gpu_launches": args.steps * (
            (len(steps_plan[0]) if pf.append_mode == "fused" else
             sum(len(st) for st in steps_plan)) + len(steps_plan) + n_combines),
    }

    if not args.no_e2e:
        # right after the timed region, so both run in the same power and
        # thermal state of the GPU (the auxiliary measurements below add
        # about a minute of load first)
        line["e2e"] = measure_e2e(args, m, w, pf, q, k, v, dev, stream, total_flops, world)
    if not args.no_append_modes:
        line["append"].update(measure_append_graph(m, w, pf, k, v, dev, hbm))
        line["append"].update(measure_fusion(args, pf, w, q, k, v, dev, stream, total_flops))
    if not args.no_graph:
        line["graph_replay"] = measure_graph(args, pf, q, k, v, dev, stream, total_flops,
                                             w.total_tokens, world)
        if pf.append_mode == "overlap" and len(steps_plan) > 1:
            line["chunk_streams"] = measure_chunk_streams(args, pf, w, q, k, v, dev, stream,
                                                          total_flops)
    if not pf.single and not args.no_graph:
        line["varlen_device_items"] = measure_varlen_dev(m, pf, w, q, dev, stream, total_flops)
    if pf.single and not args.no_projection:
        line["qkv_projection"] = measure_projection(args, m, w, pf, q, dev, stream, total_flops,
                                                    peak)
    if not args.no_last_row:
        line["last_row"] = measure_last_row(args, m, w, pf, q, dev, stream, hbm)
    if pf.mode == workloads.MODE_LBCP and pf.single and not args.no_uniform:
        # The workload's closed-form LBCP split against uniform chunks and
        # Algorithm 1's stage-1 DP (128-row units, N = 16 pipeline stages)
        # with the causal cost c (p + c / 2), Eq. 1's c (p + c), and the
        # kernel's latency model on this GPU's SM count (boundaries within 8
        # units of the closed form); all timed interleaved from CUDA graphs.
        from paper_2606_22968_gb300.pipeline import latency_balanced_bounds
        s_len, n_chunks = w.seq_lens[0], w.num_chunks[0]
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        variants = {
            "workload_boundaries": pf.bounds[0],
            "uniform_boundaries": m.mocap_lbcp_partition(s_len, n_chunks, 128,
                                                         m.MOCAP_PART_UNIFORM),
            "dp_causal_boundaries": m.mocap_lbcp_partition_dp(s_len, n_chunks, 128, 16,
                                                              m.MOCAP_COST_CAUSAL, 0),
            "dp_eq1_boundaries": m.mocap_lbcp_partition_dp(s_len, n_chunks, 128, 16,
                                                           m.MOCAP_COST_EQ1, 0),
            "dp_latency_boundaries": latency_balanced_bounds(s_len, n_chunks, w.n_q_heads,
                                                             w.n_kv_heads, w.head_dim, sms),
        }
        res = measure_partitions(w, q, k, v, dev, stream, variants)
        line["partitions"] = {"note": "each split's whole prompt and each of its chunk steps "
                                      "replayed from CUDA graphs, the splits interleaved; "
                                      "medians", "sms": sms, "dp_latency_window_units": 8,
                              **res}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        times, flops, done, threads = run_oracle_sample(
            q, k, v, pf.bounds[0], w.scale, 1, args.cpu_rows_per_chunk, 20.0)
        line["cpu_baseline"] = {
            "value": flops[0] / times[0] / 1e12, "unit": "TFLOP/s", "cores": threads,
            "kind": "oracle",
            "sample": f"up to {args.cpu_rows_per_chunk} rows x all {w.n_q_heads} heads of "
                      f"{done[0]} of {len(pf.bounds[0]) - 1} chunks (last/first alternately, "
                      f"~20 s budget): {flops[0]:.3e} FLOP in {times[0]:.1f} s, float64 oracle"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def measure_append_graph(m, w, pf, k, v, dev, hbm, reps=5, inner=10):
    """Device time of the append kernel alone, replayed from CUDA graphs (no
    launch gaps, no attention in between): the step's standalone appends
    (step 0's chunks) and, for comparison, every chunk's append as the
    unfused pipeline launches them.  Each graph holds `inner` back-to-back
    repetitions of the appends, so one graph launch's own cost is spread
    over them; the same cache rows are rewritten with the same bytes."""
    import torch
    row_bytes = w.n_kv_heads * w.head_dim * 2

    def timed(pairs):
        side = torch.cuda.Stream(dev)
        side.wait_stream(torch.cuda.current_stream(dev))
        graph = torch.cuda.CUDAGraph()

        def appends(stream):
            for r, c in pairs:
                b0, b1 = pf.bounds[r][c], pf.bounds[r][c + 1]
                base = pf.cu[r]
                m.mocap_kv_append(k[base + b0:base + b1], v[base + b0:base + b1], pf.k_cache,
                                  pf.v_cache, base + b0, stream=stream)

        with torch.cuda.stream(side):
            appends(side)  # outside the capture: one-time set-up
            with torch.cuda.graph(graph, stream=side):
                for _ in range(inner):
                    appends(side)
        torch.cuda.current_stream(dev).wait_stream(side)
        graph.replay()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            graph.replay()
        e1.record()
        torch.cuda.synchronize(dev)
        ms = e0.elapsed_time(e1) / (reps * inner)
        byts = sum(4 * (pf.bounds[r][c + 1] - pf.bounds[r][c]) * row_bytes for r, c in pairs)
        return ms, byts / (ms * 1e-3) / 1e9

    steps = pf.steps()
    ms0, gbs0 = timed(steps[0])
    ms_all, gbs_all = timed([rc for st in steps for rc in st])
    return {"kernel_ms_per_step": ms0, "kernel_gb_per_s": gbs0, "kernel_frac_of_hbm": gbs0 / hbm,
            "kernel_note": "the step's standalone appends (step 0's chunks), 10 repetitions "
                           "back to back in one CUDA graph",
            "unfused_kernel_ms_per_step": ms_all, "unfused_kernel_gb_per_s": gbs_all,
            "unfused_kernel_frac_of_hbm": gbs_all / hbm,
            "unfused_note": "every chunk's append as its own launch, 10 repetitions of the "
                            "step's appends in one graph"}


def measure_fusion(args, pf, w, q, k, v, dev, stream, total_flops, reps=3):
    """The three ways the prompt's chunk K/V reach the cache (ChunkedPrefill
    append_mode): one append launch per chunk before its attention
    ("serial"), the next chunk's append inside the attention launch
    ("fused"), or appends on a second stream beside the attention launches
    ("overlap").  Each prompt is replayed from one CUDA graph, interleaved,
    median of `reps` (no host gaps in any)."""
    import torch
    from paper_2606_22968_gb300.pipeline import APPEND_MODES, ChunkedPrefill
    times, graphs, keep = {}, {}, []
    for mode in APPEND_MODES:
        px = ChunkedPrefill(w, dev, append_mode=mode, chunk_streams=1)
        px.workspace = pf.workspace  # same split plans and scratch
        px.k_cache, px.v_cache, px.out, px.lse = pf.k_cache, pf.v_cache, pf.out, pf.lse
        px.run(q, k, v, stream)
        graphs[mode] = px.capture(q, k, v)
        times[mode] = []
        keep.append(px)
    for _ in range(reps):
        for mode, g in graphs.items():
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            g.replay()
            e0.record(stream)
            g.replay()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            times[mode].append(e0.elapsed_time(e1))
    del graphs, keep
    med = {mode: statistics.median(t) for mode, t in times.items()}
    return {"graph_ms_per_step_by_append_mode": med,
            "append_mode_used": pf.append_mode,
            "append_mode_note": "whole prompt replayed from one CUDA graph: serial = one append "
                                "launch per chunk before its attention; fused = the next chunk's "
                                "append inside the attention launch; overlap = appends on a "
                                "second stream beside the attention launches"}


def measure_chunk_streams(args, pf, w, q, k, v, dev, stream, total_flops, reps=3):
    """The prompt with its attention launches on one compute stream and
    alternating between two (ChunkedPrefill chunk_streams = 2: step i + 1 may
    use SMs that step i's last wave leaves idle), each replayed from one CUDA
    graph, interleaved, median of `reps`."""
    import torch
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    p2 = ChunkedPrefill(w, dev, append_mode="overlap", chunk_streams=2)
    p2.k_cache, p2.v_cache, p2.out, p2.lse = pf.k_cache, pf.v_cache, pf.out, pf.lse
    p2.run(q, k, v, stream)
    graphs = {1: pf.capture(q, k, v), 2: p2.capture(q, k, v)}
    times = {1: [], 2: []}
    for _ in range(reps):
        for n, g in graphs.items():
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            g.replay()
            e0.record(stream)
            g.replay()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            times[n].append(e0.elapsed_time(e1))
    del graphs, p2
    one, two = statistics.median(times[1]), statistics.median(times[2])
    return {"graph_ms_per_step_one_stream": one, "graph_ms_per_step_two_streams": two,
            "two_streams_value": total_flops / (two * 1e-3) / 1e12, "unit": "TFLOP/s",
            "note": "attention launches alternating between two compute streams "
                    "(ChunkedPrefill chunk_streams=2), appends beside them; whole prompt "
                    "replayed from one CUDA graph"}


def measure_varlen_dev(m, pf, w, q, dev, stream, total_flops, reps=5):
    """Multi-request prompts: every step's attention (chunk k of every
    request, one launch per step, caches already filled by the timed run)
    with the items as a host array and as a device array
    (mocap_chunk_attn_varlen_dev: a prepare launch before each attention
    launch, the grid sized by the step's rows), each prompt replayed from one
    CUDA graph, interleaved, median of `reps`."""
    import torch
    steps = pf.steps()
    hq, hkv, d = w.n_q_heads, w.n_kv_heads, w.head_dim
    rows = q.shape[0]
    host_items, dev_items, spaces = [], [], []
    for st in steps:
        its = [(pf.cu[r] + pf.bounds[r][c], pf.cu[r], pf.bounds[r][c],
                pf.bounds[r][c + 1] - pf.bounds[r][c]) for r, c in st]
        if len(its) == 1:
            its.append((0, 0, 0, 0))  # two items: the host form never splits either
        host_items.append(its)
        dev_items.append(torch.tensor(its, dtype=torch.int64, device=dev))
        bound = sum(x[3] for x in its)  # the step's rows: a scheduler's token budget
        need = m.mocap_chunk_attn_varlen_dev_workspace_size(len(its), bound, hq, hkv, d)
        spaces.append((torch.empty((need,), device=dev, dtype=torch.uint8), bound))
    out = torch.empty_like(pf.out)
    lse = torch.empty((hq, rows), device=dev, dtype=torch.float32)

    def host_prompt():
        for its in host_items:
            m.mocap_chunk_attn_varlen(q, pf.k_cache, pf.v_cache, its, out, lse, w.scale)

    def dev_prompt():
        for it, (ws, bound) in zip(dev_items, spaces):
            m.mocap_chunk_attn_varlen_dev(q, pf.k_cache, pf.v_cache, it, out, lse, w.scale,
                                          max_rows=bound, workspace=ws)

    graphs = {}
    for name, fn in (("host_items", host_prompt), ("device_items", dev_prompt)):
        side = torch.cuda.Stream(dev)
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            fn()
        stream.wait_stream(side)
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            fn()
        graphs[name] = g
    times = {n: [] for n in graphs}
    for _ in range(reps):
        for n, g in graphs.items():
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            g.replay()
            e0.record(stream)
            g.replay()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            times[n].append(e0.elapsed_time(e1))
    if m.mocap_last_device_status() != m.MOCAP_OK:
        raise RuntimeError("device status set in the device-item measurement")
    res = {n: statistics.median(t) for n, t in times.items()}
    return {"host_items_ms": res["host_items"], "device_items_ms": res["device_items"],
            "device_items_tflops": total_flops / (res["device_items"] * 1e-3) / 1e12,
            "note": "every step's attention launch (one compute stream, no appends), items as "
                    "a host array vs in device memory (a prepare launch per step, grid bounded "
                    "by the step's rows); prompt "
                    "replayed from one CUDA graph"}


def measure_graph(args, pf, q, k, v, dev, stream, total_flops, tokens, world):
    """The same step replayed as one captured CUDA graph (every append,
    attention launch and combine of the prompt): no per-launch host work and
    no gaps between launches.  Timed like the main region, after it.  Then
    the per-chunk latency under replay: each step's attention launch (and
    combine) as its own graph, replayed in order with events between them
    (median over `steps` passes)."""
    import torch
    graph = pf.capture(q, k, v)
    for _ in range(args.warmup):
        pf.partition()
        graph.replay()
    torch.cuda.synchronize(dev)
    barrier(world)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        pf.partition()
        graph.replay()
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, world, dev)
    del graph
    graphs = pf.capture_steps(q, k, v)
    n = len(graphs)
    per = [[] for _ in range(n)]
    for rep in range(max(3, args.steps)):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
        ev[0].record(stream)
        for i, g in enumerate(graphs):
            g.replay()
            ev[i + 1].record(stream)
        torch.cuda.synchronize(dev)
        for i in range(n):
            per[i].append(ev[i].elapsed_time(ev[i + 1]))
    pc = [statistics.median(x) for x in per]
    del graphs
    return {"ms_per_step": ms, "value": replica_throughput(total_flops, ms, world) / 1e12,
            "unit": "TFLOP/s", "prefill_tokens_per_s": replica_throughput(tokens, ms, world),
            "per_chunk_ms": {"min": min(pc), "max": max(pc), "max_over_min": max(pc) / min(pc),
                             "cv": statistics.pstdev(pc) / statistics.mean(pc),
                             "note": "each step's attention launch (and split-KV combine) as "
                                     "its own graph, replayed in order, events between replays"}}


def measure_projection(args, m, w, pf, q, dev, stream, attn_flops, peak):
    """Eq. 1's GEMM term for the same chunks: per chunk, the QKV projection of
    its hidden states (random-init weights of the model's shape) with RoPE and
    the KV append fused; then the whole chunk stage (projection, attention).
    Timed outside the main region, CUDA events, K steps after W warm-ups."""
    import torch
    hidden = args.hidden
    n_out = (w.n_q_heads + 2 * w.n_kv_heads) * w.head_dim
    gen = torch.Generator(device=dev).manual_seed(w.seed + 1000)
    x = torch.randn((w.total_tokens, hidden), generator=gen, device=dev, dtype=torch.bfloat16)
    wq = (torch.randn((n_out, hidden), generator=gen, device=dev) / hidden ** 0.5).bfloat16()
    qbuf = torch.empty_like(q)
    b = pf.bounds[0]
    gemm_flops = 2 * w.total_tokens * hidden * n_out

    def project(c):
        m.mocap_qkv_rope_append(x[b[c]:b[c + 1]], wq, qbuf[b[c]:b[c + 1]], pf.k_cache,
                                pf.v_cache, b[c], stream=stream)

    def timed(fn):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / args.steps

    n = len(b) - 1
    ms_gemm = timed(lambda: [project(c) for c in range(n)])
    ms_stage = timed(lambda: pf.run_stage(x, wq, qbuf, stream))
    ms_stage_overlap = timed(lambda: pf.run_stage(x, wq, qbuf, stream, overlap=True))
    if m.mocap_last_device_status() != m.MOCAP_OK:
        raise RuntimeError("device wait expired in the projection measurement")
    gemm_tf = gemm_flops / (ms_gemm * 1e-3) / 1e12
    line = {"hidden": hidden, "n_out": n_out, "flop_per_step": gemm_flops,
            "ms_per_step": ms_gemm, "tflops": gemm_tf, "frac_of_peak": gemm_tf / peak,
            "stage_ms_per_step": ms_stage,
            "stage_tflops": (gemm_flops + attn_flops) / (ms_stage * 1e-3) / 1e12,
            "stage_tokens_per_s": w.total_tokens / (ms_stage * 1e-3),
            # projections on their own stream, each chunk's attention waiting
            # only for its own chunk's projection (two compute streams)
            "stage_overlap_ms_per_step": ms_stage_overlap,
            "stage_overlap_tflops": (gemm_flops + attn_flops) / (ms_stage_overlap * 1e-3) / 1e12}

    # Per-chunk stage latency (projection + attention of one chunk), for the
    # workload's split and for the stage-1 DP of Algorithm 1 fed with this
    # run's measured rates: per chunk a * pairs + b * rows, i.e. in the DP's
    # doubled 128-row units k (2 s + k) + gemm_weight * k with
    # gemm_weight = 2 b / (128 a).
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill, gemm_weight, stage_balanced_bounds
    s_len, n_chunks = w.seq_lens[0], w.num_chunks[0]
    a_pair = (ms_stage - ms_gemm) * 1e-3 / (s_len * (s_len + 1) / 2)
    b_row = ms_gemm * 1e-3 / s_len

    def per_chunk_stage(pfx, reps=3):
        nx = len(pfx.bounds[0]) - 1
        times = []
        for _ in range(reps):
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(nx)]
            pfx.run_stage(x, wq, qbuf, stream, chunk_events=ev)
            torch.cuda.synchronize(dev)
            times.append([e0.elapsed_time(e1) for e0, e1 in ev])
        pc = [statistics.median(t[c] for t in times) for c in range(nx)]
        return {"min": min(pc), "max": max(pc), "max_over_min": max(pc) / min(pc),
                "cv": statistics.pstdev(pc) / statistics.mean(pc), "ms_per_step": sum(pc)}

    line["stage_per_chunk_ms"] = {"workload_split": per_chunk_stage(pf)}
    b_dp = stage_balanced_bounds(s_len, n_chunks, a_pair, b_row)
    pf_dp = ChunkedPrefill(w, dev, bounds=[b_dp])
    line["stage_per_chunk_ms"]["dp_with_gemm_term"] = {
        **per_chunk_stage(pf_dp), "gemm_weight": gemm_weight(a_pair, b_row),
        "first_chunk_rows": b_dp[1] - b_dp[0], "last_chunk_rows": b_dp[-1] - b_dp[-2]}
    del pf_dp
    if m.mocap_last_device_status() != m.MOCAP_OK:
        raise RuntimeError("device wait expired in the per-chunk stage measurement")
    return line


def measure_last_row(args, m, w, pf, q, dev, stream, hbm):
    """The one output token of a prefill-only request needs the final layer's
    attention for the last prompt row only: each request's last row against
    all its keys (memory-bound; roofline = HBM).  Uses the caches the timed
    run filled."""
    import torch
    n = len(w.seq_lens)
    rows = [pf.cu[r] for r in range(n)]
    lens = list(w.seq_lens)
    q_last = torch.stack([q[pf.cu[r] + lens[r] - 1] for r in range(n)]).contiguous()
    out = torch.empty_like(q_last)
    lse = torch.empty((w.n_q_heads, n), device=dev, dtype=torch.float32)
    ws = torch.empty((max(16, m.mocap_last_row_attn_workspace_size(lens, w.n_q_heads,
                                                                   w.n_kv_heads, w.head_dim)),),
                     device=dev, dtype=torch.uint8)
    for _ in range(args.warmup):
        m.mocap_last_row_attn(q_last, pf.k_cache, pf.v_cache, rows, lens, out, lse, w.scale,
                              workspace=ws, stream=stream)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 20
    e0.record(stream)
    for _ in range(reps):
        m.mocap_last_row_attn(q_last, pf.k_cache, pf.v_cache, rows, lens, out, lse, w.scale,
                              workspace=ws, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    if m.mocap_last_device_status() != m.MOCAP_OK:
        raise RuntimeError("device wait expired in the last-row measurement")
    us = e0.elapsed_time(e1) / reps * 1e3
    kv_bytes = sum(lens) * w.n_kv_heads * w.head_dim * 2 * 2
    gbs = kv_bytes / (us * 1e-6) / 1e9
    return {"us_per_call": us, "kv_bytes": kv_bytes, "gb_per_s": gbs, "frac_of_hbm": gbs / hbm,
            "requests": n, "note": "back-to-back calls; K/V may be partly L2-resident"}


def measure_partitions(w, q, k, v, dev, stream, variants, rounds=5):
    """Per-chunk attention latency and whole-prompt time of several chunk
    splits of one prompt (outside the timed region): each split's whole
    prompt and each of its chunk steps are captured as CUDA graphs and the
    splits are replayed interleaved, round after round (the GPU's clock under
    its power cap moves between short bursts; interleaving gives every split
    the same conditions).  Medians over the rounds."""
    import torch
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    state = {}
    for name, b in variants.items():
        px = ChunkedPrefill(w, dev, bounds=[b], chunk_streams=1)
        px.run(q, k, v, stream)
        state[name] = (px, px.capture(q, k, v), px.capture_steps(q, k, v))
    torch.cuda.synchronize(dev)
    whole = {n: [] for n in variants}
    chunks = {n: [[] for _ in range(len(b) - 1)] for n, b in variants.items()}
    names = list(variants)
    for r in range(rounds):
        for n in (names if r % 2 == 0 else names[::-1]):
            _, g, gs = state[n]
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g.replay()
            e1.record(stream)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(gs) + 1)]
            ev[0].record(stream)
            for i, gi in enumerate(gs):
                gi.replay()
                ev[i + 1].record(stream)
            torch.cuda.synchronize(dev)
            whole[n].append(e0.elapsed_time(e1))
            for i in range(len(gs)):
                chunks[n][i].append(ev[i].elapsed_time(ev[i + 1]))
    out = {}
    for n, b in variants.items():
        pc = [statistics.median(x) for x in chunks[n]]
        out[n] = {"per_chunk_attn_ms": {"min": min(pc), "max": max(pc),
                                        "max_over_min": max(pc) / min(pc),
                                        "cv": statistics.pstdev(pc) / statistics.mean(pc)},
                  "attn_ms_per_step": sum(pc), "graph_ms_per_step": statistics.median(whole[n]),
                  "first_chunk_rows": b[1] - b[0], "last_chunk_rows": b[-1] - b[-2]}
    del state
    return out


def measure_e2e(args, m, w, pf, q, k, v, dev, stream, total_flops, world):
    """The same metric through the public API with host buffers: each step
    runs ChunkedPrefill.run_from_host, which copies every chunk's Q/K/V from
    pinned host memory and its O and LSE back, overlapped with compute."""
    import torch
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    # the pipeline a user gets by default (appends beside attention, two
    # compute streams), on the timed run's buffers
    pe = ChunkedPrefill(w, dev)
    pe.k_cache, pe.v_cache, pe.out, pe.lse = pf.k_cache, pf.v_cache, pf.out, pf.lse
    pe.workspace = pf.workspace
    pf = pe
    hq, hk, hv = (t.cpu().pin_memory() for t in (q, k, v))
    ho = torch.empty(pf.out.shape, dtype=pf.out.dtype).pin_memory()
    hl = torch.empty(pf.lse.shape, dtype=pf.lse.dtype).pin_memory()
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    h2d = sum(t.numel() * t.element_size() for t in (hq, hk, hv))
    d2h = ho.numel() * ho.element_size() + hl.numel() * hl.element_size()

    def step():
        pf.partition()
        pf.run_from_host(hq, hk, hv, ho, hl, dq, dk, dv)

    # the same warm-up as the device-resident timing
    for _ in range(max(1, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    barrier(world)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    mode0 = pf.host_copies

    def timed_block(mode):
        pf.host_copies = mode
        barrier(world)
        t0.record(stream)
        for _ in range(args.e2e_steps):
            step()
        t1.record(stream)
        torch.cuda.synchronize(dev)
        barrier(world)
        return max_over_ranks(t0.elapsed_time(t1) / args.e2e_steps, world, dev)

    # blocks of single-prompt steps with the default host copies (SM copy
    # kernels, both directions) and with copy-engine copies, interleaved;
    # medians
    blocks = {mode0: [], "copy_engine": []}
    for _ in range(3):
        for mode in blocks:
            blocks[mode].append(timed_block(mode))
    pf.host_copies = mode0
    ms = statistics.median(blocks[mode0])
    ms_ce = statistics.median(blocks["copy_engine"])
    if not torch.equal(ho.to(dev), pf.out) or not torch.equal(hl.to(dev), pf.lse):
        raise RuntimeError("e2e: host copies of O / LSE differ from the device results")
    # The same steps as a stream of prompts: prompt p + 1's inputs go up while
    # prompt p computes (two device input sets), every copy still inside the
    # timed region.
    bufs = [(dq, dk, dv), (torch.empty_like(q), torch.empty_like(k), torch.empty_like(v))]
    prompts = [(hq, hk, hv, ho, hl)] * args.e2e_steps
    pf.partition()
    pf.run_prompts_from_host(prompts[:1], bufs)
    torch.cuda.synchronize(dev)
    ho.fill_(float("nan"))
    barrier(world)
    t0.record(stream)
    pf.partition()
    pf.run_prompts_from_host(prompts, bufs)
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    ms_s = max_over_ranks(t0.elapsed_time(t1) / args.e2e_steps, world, dev)
    if not torch.equal(ho.to(dev), pf.out):
        raise RuntimeError("e2e: streamed host copies of O differ from the device results")
    del bufs
    return {"value": replica_throughput(total_flops, ms, world) / 1e12, "unit": "TFLOP/s",
            "ms_per_step": ms, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "host_copies": mode0,
            "overlap": "per-chunk H2D and D2H by SM copy kernels through the pinned host pages' "
                       "device mapping, overlapped with compute (two streams, appends beside "
                       "them); ChunkedPrefill defaults",
            "blocks": "median of 3 blocks of e2e steps, interleaved with the same blocks "
                      "using copy-engine host copies",
            "copy_engine_host_copies": {"value": replica_throughput(total_flops, ms_ce, world) / 1e12,
                                    "ms_per_step": ms_ce},
            "streamed": {"value": replica_throughput(total_flops, ms_s, world) / 1e12,
                         "ms_per_step": ms_s, "prompts": args.e2e_steps,
                         "overlap": "also the next prompt's H2D under this prompt's compute"}}


def profile_case(args):
    """A single chunk_attn launch shape, repeated: the small case for ncu."""
    import torch
    import paper_2606_22968_gb300 as m
    prefix, length, hq, hkv, d = (int(x) for x in args.case.split(","))
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(7)
    q = torch.randn((length, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    kc = torch.randn((prefix + length, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    vc = torch.randn((prefix + length, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    out = torch.empty_like(q)
    lse = torch.empty((hq, length), device=dev, dtype=torch.float32)
    ws_bytes = 0
    ws = None
    if args.case_split == "auto":
        ws_bytes = m.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d)
        if ws_bytes:
            ws = torch.empty((ws_bytes,), device=dev, dtype=torch.uint8)
    ms = _repeat_timed(args, lambda: m.mocap_chunk_attn(q, kc, vc, prefix, out, lse,
                                                        1.0 / math.sqrt(d), workspace=ws))
    if m.mocap_last_device_status() != m.MOCAP_OK:
        raise RuntimeError("device wait expired")
    flops = 4 * hq * d * (length * prefix + length * (length + 1) // 2)
    print(json.dumps({"case": args.case, "ms": ms, "tflops": flops / ms / 1e9,
                      "split_workspace_bytes": ws_bytes,
                      "min_bytes": attn_min_bytes(prefix, length, hq, hkv, d)}), flush=True)
    return 0


def profile_case_append(args):
    """One KV append shape, repeated (ncu probe): rows of K and V into a cache
    of the same size."""
    import torch
    import paper_2606_22968_gb300 as m
    rows, hkv, d = (int(x) for x in args.case_append.split(","))
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(13)
    k = torch.randn((rows, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((rows, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    kc, vc = torch.empty_like(k), torch.empty_like(v)
    fn = m.mocap_kv_append_overlap if args.case_append_overlap else m.mocap_kv_append
    ms = _repeat_timed(args, lambda: fn(k, v, kc, vc, 0))
    if not (torch.equal(kc, k) and torch.equal(vc, v)):
        raise RuntimeError("append probe: cache differs from the chunk")
    byts = 2 * 2 * rows * hkv * d * 2
    print(json.dumps({"case_append": args.case_append, "overlap_kernel": args.case_append_overlap,
                      "ms": ms, "bytes": byts,
                      "gb_per_s": byts / ms / 1e6}), flush=True)
    return 0


def profile_case_host_copy(args):
    """One host <-> device copy by the SMs, repeated (ncu probe):
    'bytes,up|down,0|1' = size, direction, beside-attention form."""
    import torch
    import paper_2606_22968_gb300 as m
    nbytes, direction, beside = args.case_host_copy.split(",")
    nbytes, beside = int(nbytes), bool(int(beside))
    dev = torch.device("cuda")
    host = torch.randint(0, 256, (nbytes,), dtype=torch.uint8).pin_memory()
    devbuf = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    if direction == "up":
        ms = _repeat_timed(args, lambda: m.mocap_copy_from_host([(devbuf, host)], beside))
        ok = torch.equal(devbuf.cpu(), host)
    else:
        devbuf.copy_(host)
        back = torch.zeros(nbytes, dtype=torch.uint8).pin_memory()
        ms = _repeat_timed(args, lambda: m.mocap_copy_to_host([(back, devbuf)], beside))
        ok = torch.equal(back, host)
    if not ok:
        raise RuntimeError("host copy probe: bytes differ")
    print(json.dumps({"case_host_copy": args.case_host_copy, "ms": ms, "bytes": nbytes,
                      "gb_per_s": nbytes / ms / 1e6}), flush=True)
    return 0


def _repeat_timed(args, fn, reps=20):
    """Median over `steps` samples of the mean time of `reps` back-to-back
    calls (the host enqueues ahead of the device, so per-call host work stays
    outside the device time)."""
    import torch
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    times = []
    for _ in range(args.steps):
        ev[0].record()
        for _ in range(reps):
            fn()
        ev[1].record()
        torch.cuda.synchronize()
        times.append(ev[0].elapsed_time(ev[1]) / reps)
    return statistics.median(times)


def profile_case_qkv(args):
    """One QKV projection + RoPE + append shape, repeated (ncu probe)."""
    import torch
    import paper_2606_22968_gb300 as m
    length, hidden, hq, hkv, d = (int(x) for x in args.case_qkv.split(","))
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(11)
    x = torch.randn((length, hidden), generator=gen, device=dev, dtype=torch.bfloat16)
    w = torch.randn(((hq + 2 * hkv) * d, hidden), generator=gen, device=dev, dtype=torch.bfloat16)
    q = torch.empty((length, hq, d), device=dev, dtype=torch.bfloat16)
    kc = torch.empty((length, hkv, d), device=dev, dtype=torch.bfloat16)
    vc = torch.empty_like(kc)
    ms = _repeat_timed(args, lambda: m.mocap_qkv_rope_append(x, w, q, kc, vc, 0))
    flops = 2 * length * hidden * (hq + 2 * hkv) * d
    print(json.dumps({"case_qkv": args.case_qkv, "ms": ms, "tflops": flops / ms / 1e9}), flush=True)
    return 0


def profile_case_last_row(args):
    """One last-row attention shape, repeated (ncu probe)."""
    import torch
    import paper_2606_22968_gb300 as m
    keys, hq, hkv, d = (int(x) for x in args.case_last_row.split(","))
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(12)
    k = torch.randn((keys, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((keys, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    q = torch.randn((1, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    out = torch.empty_like(q)
    lse = torch.empty((hq, 1), device=dev, dtype=torch.float32)
    ws = torch.empty((max(16, m.mocap_last_row_attn_workspace_size([keys], hq, hkv, d)),),
                     device=dev, dtype=torch.uint8)
    ms = _repeat_timed(args, lambda: m.mocap_last_row_attn(q, k, v, [0], [keys], out, lse,
                                                           1.0 / math.sqrt(d), workspace=ws))
    byts = keys * hkv * d * 4
    print(json.dumps({"case_last_row": args.case_last_row, "ms": ms,
                      "gb_per_s": byts / ms / 1e6}), flush=True)
    return 0


def main():
    args = parse_args()
    if args.case:
        return profile_case(args)
    if args.case_append:
        return profile_case_append(args)
    if args.case_host_copy:
        return profile_case_host_copy(args)
    if args.case_qkv:
        return profile_case_qkv(args)
    if args.case_last_row:
        return profile_case_last_row(args)
    rank, world, local = init_dist(args)
    try:
        if args.impl == "reference":
            return reference_arm(args, rank, world)
        return ours_arm(args, rank, world, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
