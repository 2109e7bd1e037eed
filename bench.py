"""Benchmark of the HSA hot path on one GB300 (or N independent replicas).

One step = one pass of the whole hot path over one synthetic HSA layer:
  partition (once) and then, for each measured iteration i, active set ->
  gather of the active hidden rows -> KV-cache scatter -> active attention ->
  cached Euler.
Default workload: Wan-2.1-1.3B shaped layer, N = 32760 tokens (21x30x52
grid), 12 heads x 128, bf16, groups 25%@40 + 25%@20 + 50%@10 of T = 40, the
three iterations i = 0, 2, 1 (100%, 50%, 25% active).

value  = active-attention FLOPs (4 |A| N D H summed over the step) / step
         time, TFLOP/s, whole job (all replicas); inputs resident in HBM,
         L2 flushed between steps, CUDA events on the launching stream.
e2e    = the same metric through the C ABI with host buffers: the step's
         inputs (statistic, compact Q/K/V and velocities of each iteration's
         active tokens) are copied from pinned host memory and the attention
         outputs and the latent are read back inside the timed region.
--impl reference times the CPU oracle (the reference implementation here) on
a bounded sample of the same workload, on the host cores.

Multi-GPU: the path is run as independent replicas (one per GPU, no
collective on the data path); the timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import concurrent.futures as cf
import dataclasses
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

import synth  # noqa: E402

METRIC = "HSA active-attention TFLOP/s vs BF16 peak; KV-sync/Euler HBM GB/s"
# The largest workload that fits one GPU: the full 40-iteration schedule of the
# 720p Wan-14B layer.  The others run briefly after it (config.also).
HEADLINE = "wan14b_720p"
ALSO = ("wan13b", "wan14b_boxes", "ltx", "tiny_f32")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20
HEAD_START_CYCLES = 6_000_000      # ~3 ms of GPU spin while the host enqueues a timed step


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="hsa", choices=["hsa", "reference"])
    p.add_argument("--workload", default=HEADLINE, choices=list(synth.WORKLOADS))
    p.add_argument("--heads", type=int, default=0,
                   help="override the workload's head count (small cases for ncu captures)")
    p.add_argument("--iters", default="",
                   help="override the measured iterations, e.g. 0,4,2,1")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-also", action="store_true",
                   help="skip the short runs of the other workloads (config.also)")
    p.add_argument("--memory-sweep", action="store_true",
                   help="HBM size sweep of gather, KV scatter and cached Euler (L2 flushed)")
    return p.parse_args()


def workload_of(args) -> synth.Workload:
    w = synth.WORKLOADS[args.workload]
    if args.heads:
        w = dataclasses.replace(w, H=args.heads)
    if args.iters:
        w = dataclasses.replace(w, iters=tuple(int(x) for x in args.iters.split(",")))
    return w


# ------------------------------------------------------------ distributed

def dist_setup(backend):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group(backend=backend)
        return dist, dist.get_rank(), ws, int(os.environ.get("LOCAL_RANK", "0"))
    return None, 0, 1, 0


def max_over_ranks(dist, value: float, device) -> float:
    if dist is None:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist):
    if dist is not None:
        dist.barrier()


# ------------------------------------------------------------ peaks/clocks

def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle samples every 200 ms during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, local_rank: int):
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        ids = [v.strip() for v in vis.split(",")] if vis else []
        self.gpu = ids[local_rank] if local_rank < len(ids) else str(local_rank)
        self.proc = None
        self.path = os.path.join("/tmp", f"hsa_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
            # nvidia-smi's start-up (driver and NVML initialisation) can hold
            # the GPU for a moment: start timing only once it has written its
            # first sample (at most 10 s)
            t0 = time.time()
            while time.time() - t0 < 10.0 and self.proc.poll() is None:
                time.sleep(0.05)
                if os.path.getsize(self.path) > 0:
                    break
            time.sleep(0.25)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None:
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[5:9]))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[3])
                          if v.lower() == "active"})
        loaded = [r[0] for r in rows if r[2] > 200.0] or [r[0] for r in rows]
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------- workload

def host_inputs(w: synth.Workload, rep: int = 0):
    """The workload's seeded host tensors: hidden rows, Q, K/V cache, fresh K/V,
    latent, velocity cache, fresh velocities (multi-GB shapes drawn in blocks
    on the host cores, synth.normal_blocks)."""
    seed = lambda t: synth.seed_for(w.cid, rep, t)  # noqa: E731
    dt = w.dtype
    N, H, D, C = w.N, w.H, w.D, w.C
    big = lambda shape, t: synth.normal_blocks(shape, seed(t), dt)  # noqa: E731
    return {"hidden": big((N, H * D), 1), "q": big((N, H, D), 2), "kc": big((N, H, D), 3),
            "vc": big((N, H, D), 4), "kf": big((N, H, D), 5), "vf": big((N, H, D), 6),
            "x": synth.normal((N, C), seed(7)), "vh": synth.normal((N, C), seed(8)),
            "v_fresh": synth.normal((N, C), seed(9))}


class Layer:
    """Resident device state and inputs of one HSA layer workload."""

    def __init__(self, w: synth.Workload, dev, rep: int = 0, keep_host: bool = False):
        self.w, self.dev = w, dev
        N, H, D = w.N, w.H, w.D
        self.stat_h, self.counts = synth.stat_for(w, rep)
        host = host_inputs(w, rep)
        self.host = host if keep_host else None
        self.stat = self.stat_h.to(dev)
        for k, t in host.items():
            setattr(self, k, t.to(dev))
        self.group_of = torch.empty(N, dtype=torch.int32, device=dev)
        self.idx = torch.empty(N, dtype=torch.int32, device=dev)
        self.pos = torch.empty(N, dtype=torch.int32, device=dev)
        self.gathered = torch.empty((N, H * D), dtype=self.hidden.dtype, device=dev)
        self.out = torch.empty((N, H, D), dtype=self.q.dtype, device=dev)
        self.iters = list(w.iters)


def algorithmic(w, n_act):
    """Algorithmic FLOPs / bytes per launch of each kernel (see design notes)."""
    N, H, D, C = w.N, w.H, w.D, w.C
    eb = 2 if w.dtype == "bf16" else 4
    row = H * D * eb
    return {
        "attention_flops": 4.0 * n_act * N * D * H,
        "attention_bytes": (2 * n_act + 2 * N) * H * D * eb + 4 * n_act,
        "gather": n_act * (2 * row + 4),
        "scatter": n_act * (4 * row + 4),
        "euler": (N - n_act) * 12 * C + n_act * 16 * C + 4 * N,
        "active": 4 * N + 4 * n_act + 4 * N,
    }


def representative_iters(w, counts):
    """First iteration of each distinct active-set size, in schedule order
    (the CPU legs' sample of the schedule)."""
    import oracle
    seen, out = set(), []
    for it in w.iters:
        n = oracle.active_count(w.budgets, counts, w.T, it, w.window_pct)
        if n not in seen:
            seen.add(n)
            out.append(it)
    return out


# ---------------------------------------------------------------- hsa arm

def run_hsa(args, dist, rank, world, local_rank):
    import paper_2605_06892_gb300 as hsa
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    w = workload_of(args)
    want_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    L = Layer(w, dev, keep_host=want_cpu)
    peaks, peak_src = load_peaks()
    res = measure(args, hsa, L, dev, dist, world, local_rank, args.steps, peaks)
    flops_step, ms_per_step = res["flops_step"], res["ms_per_step"]
    value = world * flops_step / (ms_per_step * 1e-3) / 1e12
    kernels = res["kernels"]
    att_tflops = kernels["attention"]["tflops"]
    clocks = res["clocks"]
    # Peak for the roofline: the measured burst figure for a kernel that runs in
    # short steps, the sustained one (seconds-long loop under the power cap) for
    # a kernel timed inside a step that keeps the GPU busy for about a second.
    long_step = ms_per_step >= 500.0
    peak = peaks["bf16_tflops_sustained"] if long_step else peaks["bf16_tflops"]
    roofline = {
        "bound": "tensor", "achieved": att_tflops, "peak": peak, "unit": "TFLOP/s",
        "frac": att_tflops / peak, "traffic": profiled_traffic(w, res["n_of"]),
        "peak_source": (f"{peak_src} bf16 sustained (kernel timed inside a "
                        f"{ms_per_step / 1e3:.2f} s step)" if long_step
                        else f"{peak_src} bf16 burst"),
        "frac_burst": att_tflops / peaks["bf16_tflops"],
        "frac_sustained": att_tflops / peaks["bf16_tflops_sustained"],
        "clock_normalised": clock_normalised(att_tflops, clocks, peaks),
    }
    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) Q/K/V, lognormal statistic; no model weights)",
        "config": {"workload": workload_desc(w, L.counts),
                   "iterations": res["iterations"], "parallelism": f"replicas x{world}",
                   "l2": "flushed (256 MiB write) between steps; K/V cache and Q exceed L2",
                   "q_load": "index-driven (q_idx into the [N,H,D] query tensor)"},
        "kernels": kernels, "roofline": roofline, "dense_baseline": res["dense_baseline"],
        "timing": res["timing"],
        "gpu_launches": res["launches"],
        "clocks": clocks,
    }
    if not args.no_e2e:
        line["e2e"] = run_e2e(args, hsa, L, res["sig"], res["n_of"], torch.cuda.current_stream(dev),
                              dev, dist, world, flops_step, local_rank)
    if want_cpu:
        line["cpu_baseline"] = cpu_baseline(w, L)
    with_also = (not args.no_also and not args.heads and not args.iters
                 and args.workload == HEADLINE)
    also = {}
    if with_also:
        # The same layer and inputs with the HSA-50 preset's caching window
        # (k = 80 %: the first and last m = 4 iterations are full passes).
        wk = dataclasses.replace(w, name=w.name + "_window80", window_pct=80)
        L.w = wk
        steps = max(3, min(args.steps, 10))
        also[wk.name] = also_summary(
            wk, L.counts, steps, measure(args, hsa, L, dev, dist, world, local_rank, steps,
                                         peaks), peaks, world)
    host = L.host
    del L, host
    torch.cuda.empty_cache()
    if with_also:
        also.update(run_also(args, hsa, dev, dist, world, local_rank, peaks))
        line["config"]["also"] = also
    if rank == 0:
        print(json.dumps(line), flush=True)


def measure(args, hsa, L, dev, dist, world, local_rank, steps, peaks):
    """Warm-up, then `steps` timed steps of the workload's hot path (CUDA
    events on the launching stream, L2 flushed between steps, clocks sampled),
    then the dense all-token iteration.  Returns the per-kernel and per-step
    figures."""
    w = L.w
    T, budgets = w.T, w.budgets
    sig = hsa.hsa_sigma_schedule(T, w.shift)
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(w.N), dtype=torch.uint8, device=dev)
    ws_att = torch.empty(max(1, hsa.hsa_active_attention_workspace_bytes(
        w.N, w.N, w.H, w.D, 0 if w.dtype == "bf16" else 1)), dtype=torch.uint8, device=dev)
    L.ws_att = ws_att
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    n_of = {it: hsa.hsa_active_count(budgets, L.counts, T, it, w.window_pct) for it in L.iters}

    kinds = ("partition", "active", "gather", "scatter", "attention", "euler")

    def step(record, strm=None):
        """One pass of the hot path; record(kind, fn) launches fn between events.
        Launches on `strm` (default: the benchmark's stream)."""
        st = strm if strm is not None else stream
        record("partition", lambda: hsa.hsa_partition(L.stat, T, budgets, L.counts, L.group_of,
                                                      ws, st))
        for it in L.iters:
            n = n_of[it]
            ds = sig[it + 1] - sig[it]
            record("active", lambda: hsa.hsa_partition_active(L.group_of, T, budgets, it, L.idx,
                                                              L.pos, w.window_pct, st))
            record("gather", lambda: hsa.hsa_gather_active(L.hidden, L.idx, n, L.gathered, st))
            record("scatter", lambda: hsa.hsa_kv_sync_scatter(L.kc, L.vc, L.kf, L.vf, L.idx, n,
                                                              st))
            record("attention", lambda: hsa.hsa_active_attention(L.q, L.idx, n, L.kc, L.vc,
                                                                 L.out, 0.0, ws_att, st))
            record("euler", lambda: hsa.hsa_cached_euler(L.x, L.vh, L.v_fresh, L.pos, ds, n, st))

    plain = lambda kind, fn: fn()  # noqa: E731
    for _ in range(args.warmup):
        flush.zero_()
        step(plain)
    torch.cuda.synchronize()
    assert hsa.hsa_get_device_error(stream) == 0

    per_kernel = {k: [] for k in kinds}
    step_events, bd_events = [], []

    def timed(kind, fn):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        per_kernel[kind].append((a, b))

    def one_step(record, events):
        flush.zero_()                           # L2 flush, outside the step's events
        # The GPU spins for a moment (outside the events) while the host enqueues
        # the step, so that host launch latency does not open gaps between the
        # step's kernels: the events time the device's work.  (The e2e leg keeps
        # the host in the loop.)
        torch.cuda._sleep(HEAD_START_CYCLES)
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        step(record)
        s1.record(stream)
        events.append((s0, s1))

    # The timed steps carry no event inside them (an event between two kernels
    # keeps the second from starting during the first's last moments, which
    # costs a few microseconds per launch on short steps).  The per-kernel
    # breakdown comes from separate steps with an event pair around every call.
    bsteps = max(2, min(steps, 5))
    barrier(dist)
    torch.cuda.synchronize()
    launches0 = hsa.hsa_launch_count()
    with ClockSampler(local_rank) as clocks:
        for _ in range(steps):
            one_step(plain, step_events)
        torch.cuda.synchronize()
        launches = hsa.hsa_launch_count() - launches0       # this library's kernels only
        barrier(dist)
        for _ in range(bsteps):
            one_step(timed, bd_events)
        torch.cuda.synchronize()
    step_ms = [a.elapsed_time(b) for a, b in step_events]
    total_ms = max_over_ranks(dist, sum(step_ms), dev)
    ms_per_step = total_ms / steps
    bd_ms_per_step = sum(a.elapsed_time(b) for a, b in bd_events) / bsteps
    kern_ms = {k: sum(a.elapsed_time(b) for a, b in v) / bsteps for k, v in per_kernel.items()}
    status = hsa.hsa_get_device_error(stream)
    assert status == 0, f"device error {status}"

    flops_step = sum(algorithmic(w, n_of[it])["attention_flops"] for it in L.iters)
    bytes_step = {k: sum(algorithmic(w, n_of[it])[k] for it in L.iters)
                  for k in ("gather", "scatter", "euler", "active")}
    kernels = {
        "attention": {"ms": kern_ms["attention"],
                      "tflops": flops_step / (kern_ms["attention"] * 1e-3) / 1e12},
        "partition": {"ms": kern_ms["partition"]},
    }
    for k in ("gather", "scatter", "euler", "active"):
        gbs = bytes_step[k] / (kern_ms[k] * 1e-3) / 1e9
        kernels[k] = {"ms": kern_ms[k], "gbs": gbs, "frac_hbm": gbs / peaks["hbm_gbs"]}
    # per-iteration layer time (the five kernels of each iteration), and the
    # same iteration with every token active (i = 0 activates every group):
    # the dense all-token baseline, through the same kernels
    n_it = len(L.iters)
    it_ms = [0.0] * n_it
    att_ms = [0.0] * n_it
    for kind in ("active", "gather", "scatter", "attention", "euler"):
        for e, (a, b) in enumerate(per_kernel[kind]):
            t = a.elapsed_time(b) / bsteps
            it_ms[e % n_it] += t
            if kind == "attention":
                att_ms[e % n_it] += t
    graph = graph_replay(args, hsa, step, plain, flush, stream, steps)
    dense = dense_iteration(args, hsa, L, sig, flush, ws_att, stream)
    by_frac = {}
    for m, it in enumerate(L.iters):
        f = round(n_of[it] / w.N, 4)
        d = by_frac.setdefault(f, {"n_active": n_of[it], "iterations": [], "ms": [],
                                   "attention_ms": []})
        d["iterations"].append(it)
        d["ms"].append(it_ms[m])
        d["attention_ms"].append(att_ms[m])
    iterations = {}
    for f, d in sorted(by_frac.items(), reverse=True):
        ms = statistics.mean(d["ms"])
        iterations[f"{f:g}"] = {
            "n_active": d["n_active"], "iterations": d["iterations"], "ms": ms,
            "attention_ms": statistics.mean(d["attention_ms"]), "vs_dense": ms / dense["ms"]}
    dense_baseline = {
        "iteration_ms": dense["ms"], "attention_ms": dense["attention_ms"],
        "step_ms_all_dense": n_it * dense["ms"] + kern_ms["partition"],
        "step_vs_all_dense": ms_per_step / (n_it * dense["ms"] + kern_ms["partition"]),
        "ideal_vs_all_dense": sum(n_of.values()) / (n_it * w.N),
        "what": f"{n_it} iterations with every token active (same kernels, |A| = N), "
                "against the measured step; L2 flushed before each dense iteration"}
    kern_sum = sum(kern_ms.values())
    timing = {"step_ms": ms_per_step, "breakdown_steps": bsteps,
              "breakdown_step_ms": bd_ms_per_step, "kernels_sum_ms": kern_sum,
              "gaps_ms": bd_ms_per_step - kern_sum, "graph_ms_per_step": graph,
              "what": "step_ms: the timed steps (no event inside a step); breakdown_step_ms: "
                      "separate steps with an event pair around every call, whose per-kernel "
                      "times sum to kernels_sum_ms (gaps_ms: the rest of those steps); "
                      "graph_ms_per_step: the same step captured once in a CUDA graph and "
                      "replayed.  L2 flushed before every step; each step is enqueued while "
                      "the GPU spins (outside the events), so host launch latency does not "
                      "appear inside a step"}
    return {"flops_step": flops_step, "ms_per_step": ms_per_step, "kernels": kernels,
            "iterations": iterations, "dense_baseline": dense_baseline, "launches": launches,
            "clocks": clocks.summary(), "sig": sig, "n_of": n_of, "timing": timing}


def graph_replay(args, hsa, step, plain, flush, stream, steps):
    """The step captured once in a CUDA graph and replayed: the device time of
    the same launches without the host's launch gaps.  The library does its host
    work (argument checks, tensor maps, the tail plan) before enqueueing, so the
    replay runs exactly the kernels of an eager step.  Returns ms per replay."""
    reps = max(2, min(steps, 5))
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step(plain, torch.cuda.current_stream())     # the capture stream
    g.replay()                                   # warm-up replay
    torch.cuda.synchronize()
    tot = 0.0
    for _ in range(reps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        tot += a.elapsed_time(b)
    assert hsa.hsa_get_device_error(stream) == 0
    del g
    return tot / reps


def clock_normalised(att_tflops, clocks, peaks):
    """The attention rate against the cuBLAS denominator at equal SM clock, and
    against the tensor pipe's own rate (8192 bf16 FLOP per clock per SM, dense)
    at the sampled clock.  The denominators' clock: the median SM clock the
    peak measurement saw under load (MEASURED_PEAKS.json), which the seconds-
    long sustained loop dominates."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            peak_mhz = float(json.load(f)["clocks_under_load"]["sm_mhz_median"])
    except (OSError, KeyError, ValueError, TypeError):
        peak_mhz = None
    if not clocks or not clocks.get("sm_mhz"):
        return None
    mhz = clocks["sm_mhz"]
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    out = {"sm_mhz": mhz, "tensor_pipe_peak_tflops_at_clock": 8192 * sms * mhz * 1e6 / 1e12}
    out["frac_of_tensor_pipe_at_clock"] = att_tflops / out["tensor_pipe_peak_tflops_at_clock"]
    if peak_mhz:
        out["cublas_sustained_sm_mhz"] = peak_mhz
        out["frac_of_cublas_sustained_at_equal_clock"] = (
            (att_tflops / mhz) / (peaks["bf16_tflops_sustained"] / peak_mhz))
    return out


def run_also(args, hsa, dev, dist, world, local_rank, peaks):
    """Short runs of the other workloads (no e2e, no CPU leg): their step rate,
    attention rate and roofline fraction, memory-kernel fractions and the
    iteration time against the dense iteration."""
    out = {}
    for name in ALSO:
        w = synth.WORKLOADS[name]
        L = Layer(w, dev)
        steps = max(3, min(args.steps, 10))
        res = measure(args, hsa, L, dev, dist, world, local_rank, steps, peaks)
        out[name] = also_summary(w, L.counts, steps, res, peaks, world)
        del L
        torch.cuda.empty_cache()
    return out


def also_summary(w, counts, steps, res, peaks, world):
    """The figures `config.also` gives for one extra workload run."""
    att = res["kernels"]["attention"]["tflops"]
    return {
        "workload": workload_desc(w, counts), "steps": steps,
        "ms_per_step": res["ms_per_step"],
        "value": world * res["flops_step"] / (res["ms_per_step"] * 1e-3) / 1e12,
        "attention_tflops": att,
        "attention_frac_burst": att / peaks["bf16_tflops"] if w.dtype == "bf16" else None,
        "gather_frac_hbm": res["kernels"]["gather"]["frac_hbm"],
        "scatter_frac_hbm": res["kernels"]["scatter"]["frac_hbm"],
        "euler_frac_hbm": res["kernels"]["euler"]["frac_hbm"],
        "partition_ms": res["kernels"]["partition"]["ms"],
        "iterations_vs_dense": {f: d["vs_dense"] for f, d in res["iterations"].items()},
        "step_vs_all_dense": res["dense_baseline"]["step_vs_all_dense"],
        "ideal_vs_all_dense": res["dense_baseline"]["ideal_vs_all_dense"],
        "graph_ms_per_step": res["timing"]["graph_ms_per_step"],
        "gpu_launches": res["launches"], "clocks": res["clocks"]}


def dense_iteration(args, hsa, L, sig, flush, ws_att, stream, reps=None):
    """Time one HSA iteration with every token active (iteration 0 of the
    schedule activates every group): active set, gather, KV-sync scatter,
    attention over all N queries, cached Euler.  L2 flushed before each rep;
    outside the benchmark's timed region."""
    w = L.w
    T, budgets = w.T, w.budgets
    reps = reps or max(3, min(args.steps, 10))
    ds = sig[1] - sig[0]
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    tot, att = [], []
    for r in range(reps + 1):
        flush.zero_()
        torch.cuda._sleep(HEAD_START_CYCLES)
        a, b, c, d = ev(), ev(), ev(), ev()
        a.record(stream)
        hsa.hsa_partition_active(L.group_of, T, budgets, 0, L.idx, L.pos, w.window_pct, stream)
        hsa.hsa_gather_active(L.hidden, L.idx, w.N, L.gathered, stream)
        hsa.hsa_kv_sync_scatter(L.kc, L.vc, L.kf, L.vf, L.idx, w.N, stream)
        b.record(stream)
        hsa.hsa_active_attention(L.q, L.idx, w.N, L.kc, L.vc, L.out, 0.0, ws_att, stream)
        c.record(stream)
        hsa.hsa_cached_euler(L.x, L.vh, L.v_fresh, L.pos, ds, w.N, stream)
        d.record(stream)
        if r > 0:                                  # the first rep is a warm-up
            tot.append((a, d))
            att.append((b, c))
    torch.cuda.synchronize()
    assert hsa.hsa_get_device_error(stream) == 0
    return {"ms": sum(x.elapsed_time(y) for x, y in tot) / reps,
            "attention_ms": sum(x.elapsed_time(y) for x, y in att) / reps}


def run_e2e(args, hsa, L, sig, n_of, stream, dev, dist, world, flops_step, local_rank=0):
    """Same step through the C ABI with host buffers (pinned).  Copies run on
    their own streams and overlap the kernels: each iteration's inputs are
    copied in two iterations ahead into a ring of three device buffers (so a
    large copy can overlap more than one short iteration; the next step's first
    iterations are copied in during this step's last ones), each attention
    output is copied out as soon as it is ready, and the latent after the step.
    Timed from the first host-to-device copy to the last device-to-host copy."""
    w = L.w
    T, budgets = w.T, w.budgets
    iters = L.iters
    n_max = max(n_of.values())
    pin = lambda t: t.cpu().pin_memory()  # noqa: E731
    h_stat = pin(L.stat)
    h_q, h_kf, h_vf = pin(L.q[:n_max]), pin(L.kf[:n_max]), pin(L.vf[:n_max])
    h_vfr = pin(L.v_fresh[:n_max])
    h_out = [torch.empty((n_of[it], w.H, w.D), dtype=L.out.dtype).pin_memory() for it in iters]
    h_x = torch.empty_like(L.x, device="cpu").pin_memory()
    ahead = min(2, len(iters))           # iterations whose inputs are copied in ahead
    nbuf = ahead + 1
    bufs = [dict(q=torch.empty_like(L.q[:n_max]), kf=torch.empty_like(L.kf[:n_max]),
                 vf=torch.empty_like(L.vf[:n_max]), vfr=torch.empty_like(L.v_fresh[:n_max]))
            for _ in range(nbuf)]
    outs = [torch.empty((n_max, w.H, w.D), dtype=L.out.dtype, device=dev) for _ in range(2)]
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(w.N), dtype=torch.uint8, device=dev)
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    h2d = L.stat.numel() * 4
    d2h = h_x.numel() * 4
    for it in iters:
        n = n_of[it]
        h2d += n * w.H * w.D * 2 * 3 + n * w.C * 4
        d2h += n * w.H * w.D * 2
    ev = lambda: torch.cuda.Event()  # noqa: E731
    # slot events persist across steps: input slot j % nbuf is free for the
    # copy-in of use j once compute of use j - nbuf is done (in_free); output
    # buffer j % 2 once the copy-out of use j - 2 is done (out_free)
    st = {"j": 0, "in_free": [None] * nbuf, "out_free": [None, None], "stat_free": None,
          "x_free": None}

    n_it = len(iters)

    def step(prefetch_next):
        """One step; with prefetch_next the copies of the next step's first
        `ahead` iterations are issued during this step's last iterations."""
        j0 = st["j"]
        loaded = st.pop("pending", {})
        with torch.cuda.stream(s_in):
            if st["stat_free"] is not None:
                s_in.wait_event(st["stat_free"])
            L.stat.copy_(h_stat, non_blocking=True)
            stat_ready = ev()
            stat_ready.record(s_in)

        def load(k):
            """Copy in the inputs of use j0 + k: iteration k of this step, or
            (k >= n_it) iteration k - n_it of the next step."""
            j = j0 + k
            b, n = bufs[j % nbuf], n_of[iters[k % n_it]]
            with torch.cuda.stream(s_in):
                if st["in_free"][j % nbuf] is not None:
                    s_in.wait_event(st["in_free"][j % nbuf])
                b["q"][:n].copy_(h_q[:n], non_blocking=True)
                b["kf"][:n].copy_(h_kf[:n], non_blocking=True)
                b["vf"][:n].copy_(h_vf[:n], non_blocking=True)
                b["vfr"][:n].copy_(h_vfr[:n], non_blocking=True)
                e = ev()
                e.record(s_in)
            return e

        for k in range(ahead):
            if k not in loaded:
                loaded[k] = load(k)
        stream.wait_event(stat_ready)
        hsa.hsa_partition(L.stat, T, budgets, L.counts, L.group_of, ws, stream)
        st["stat_free"] = ev()
        st["stat_free"].record(stream)
        for k, it in enumerate(iters):
            if k + ahead < n_it:
                loaded[k + ahead] = load(k + ahead)
            elif prefetch_next:
                st.setdefault("pending", {})[k + ahead - n_it] = load(k + ahead)
            j = j0 + k
            b, n = bufs[j % nbuf], n_of[it]
            ds = sig[it + 1] - sig[it]
            stream.wait_event(loaded[k])
            if st["out_free"][j % 2] is not None:
                stream.wait_event(st["out_free"][j % 2])
            hsa.hsa_partition_active(L.group_of, T, budgets, it, L.idx, L.pos, w.window_pct,
                                     stream)
            hsa.hsa_gather_active(L.hidden, L.idx, n, L.gathered, stream)
            hsa.hsa_kv_sync_scatter(L.kc, L.vc, b["kf"], b["vf"], L.idx, n, stream)
            out = outs[j % 2]
            hsa.hsa_active_attention(b["q"], None, n, L.kc, L.vc, out, 0.0, L.ws_att, stream)
            e_att = ev()
            e_att.record(stream)
            if k == 0 and st["x_free"] is not None:
                stream.wait_event(st["x_free"])          # previous latent copied out
            hsa.hsa_cached_euler(L.x, L.vh, b["vfr"], L.pos, ds, n, stream)
            st["in_free"][j % nbuf] = ev()
            st["in_free"][j % nbuf].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(e_att)
                h_out[k].copy_(out[:n], non_blocking=True)
                st["out_free"][j % 2] = ev()
                st["out_free"][j % 2].record(s_out)
        st["j"] = j0 + len(iters)
        fin = ev()
        fin.record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(fin)
            h_x.copy_(L.x, non_blocking=True)
            st["x_free"] = ev()
            st["x_free"].record(s_out)

    # Every step's inputs are copied inside the timed region exactly once: the
    # warm-up steps prefetch nothing, and the last timed step does not copy in
    # the inputs of a step that will not run.
    for _ in range(args.warmup):
        step(False)
    torch.cuda.synchronize()
    barrier(dist)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local_rank) as clocks:
        a.record(s_in)
        stream.wait_event(a)
        s_out.wait_event(a)
        for i in range(args.steps):
            step(i + 1 < args.steps)
        s_out.wait_stream(stream)
        s_out.wait_stream(s_in)
        b.record(s_out)
        torch.cuda.synchronize()
    barrier(dist)
    ms = max_over_ranks(dist, a.elapsed_time(b), dev) / args.steps
    assert hsa.hsa_get_device_error(stream) == 0
    return {"value": world * flops_step / (ms * 1e-3) / 1e12, "unit": "TFLOP/s",
            "ms_per_step": ms, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "copies": "pinned host buffers; inputs copied two iterations ahead (across "
                      "the step boundary too) on a copy stream, outputs copied back on "
                      "another, overlapping the kernels",
            "q_load": "compact (the caller copies the active rows' Q; q_idx = NULL)",
            "clocks": clocks.summary()}


def code_digest(text: str) -> str:
    """Digest of a CUDA source with its comments and whitespace removed, so
    that an edit to comments alone does not invalidate a profile."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    text = " ".join(text.split())
    return hashlib.sha256(text.encode()).hexdigest()[:16]


def profiled_traffic(w, n_of):
    """DRAM bytes per attention launch (read + write), averaged over the step's
    launches, from the committed ncu summary of this workload's attention
    kernel, if it was taken on the current attention code (comments aside);
    else None.  The summary lists bytes per launch at each active fraction,
    per head (`traffic_per_head_bytes <frac>: <bytes>`), measured on a case
    with fewer heads; heads are independent, so a launch's traffic scales with
    H."""
    path = os.path.join(ROOT, "profiles", f"attention_{w.name}.md")
    src = os.path.join(ROOT, "paper_2605_06892_gb300", "csrc", "hsa_attention.cu")
    try:
        digest = code_digest(open(src).read())
        per_head, sha = {}, None
        for line in open(path):
            if line.startswith("code_sha256:"):
                sha = line.split(":", 1)[1].strip()
            elif line.startswith("traffic_per_head_bytes"):
                k, v = line.split(":", 1)
                per_head[round(float(k.split()[1]), 4)] = float(v)
        if sha != digest or not per_head:
            return None
        tot = 0.0
        for it, n in n_of.items():
            f = round(n / w.N, 4)
            if f not in per_head:
                return None
            tot += per_head[f] * w.H
        return tot / len(n_of)
    except (OSError, KeyError, ValueError, IndexError):
        return None


# ----------------------------------------------------------- CPU oracle leg

def host_cores() -> int:
    return max(1, len(os.sched_getaffinity(0)))


def _oracle_sample(w, stat, counts, t, rows_per_iter, iters, threads):
    """The oracle's pass over one bounded sample of the workload: partition,
    then for each iteration in `iters` the active set, gather, KV scatter and
    cached Euler at full size, and attention of `rows_per_iter` active query
    rows (all heads, all N keys).  With threads > 1 the same oracle calls run
    on disjoint slices (rows of the gather and scatter, tokens of the Euler
    step, query rows of the attention) in a thread pool; ctypes releases the
    GIL during each call.  Returns (seconds, attention FLOPs done)."""
    import oracle
    sig = oracle.sigmas(w.T, w.shift)
    pool = cf.ThreadPoolExecutor(max_workers=threads) if threads > 1 else None

    def run(fn, parts):
        if pool is None:
            for p in parts:
                fn(p)
        else:
            list(pool.map(fn, parts))

    def cuts(n):
        k = max(1, min(threads, n))
        return [(n * i // k, n * (i + 1) // k) for i in range(k)]

    t0 = time.perf_counter()
    g = oracle.partition(stat, w.T, w.budgets, counts)
    flops = 0.0
    for it in iters:
        idx, pos = oracle.active_set(g, w.T, w.budgets, it, w.window_pct)
        n = idx.numel()
        run(lambda c: oracle.gather(t["hidden"], idx[c[0]:c[1]]), cuts(n))
        run(lambda c: oracle.kv_scatter(t["kc"], t["vc"], t["kf"][c[0]:c[1]],
                                        t["vf"][c[0]:c[1]], idx[c[0]:c[1]]), cuts(n))
        rows = idx[:rows_per_iter]
        run(lambda c: oracle.attention(t["q"], t["kc"], t["vc"], q_idx=rows[c[0]:c[1]]),
            cuts(rows.numel()))
        flops += 4.0 * rows.numel() * w.N * w.D * w.H
        ds = float(sig[it + 1] - sig[it])
        vfr = t["v_fresh"][:n]
        run(lambda c: oracle.cached_euler_f32(t["x"][c[0]:c[1]], t["vh"][c[0]:c[1]], vfr,
                                              pos[c[0]:c[1]], ds), cuts(w.N))
    el = time.perf_counter() - t0
    if pool is not None:
        pool.shutdown()
    return el, flops


def _sample_text(w, rows, iters, threads, secs):
    return (f"partition, then for iterations {iters} (one per distinct active-set size of "
            f"the schedule) active set, gather, KV scatter and cached Euler at full size "
            f"plus attention of {rows} active query rows x {w.H} heads x {w.N} keys per "
            f"iteration; fp64 oracle, {threads} thread(s), {secs:.1f} s")


def cpu_baseline(w, L, target_mt_s=10.0):
    """The oracle timed on the host cores on a bounded sample of the workload:
    all cores (the oracle's own calls on disjoint slices in a thread pool) and,
    beside it, a single thread on the schedule's first iteration."""
    counts = L.counts
    t = L.host
    stat = L.stat_h
    iters = representative_iters(w, counts)
    cores = host_cores()
    st_t, st_f = _oracle_sample(w, stat, counts, t, 1, iters[:1], 1)
    # st_t bounds one query row's time from above (it includes the full-size
    # gather, scatter and Euler of the iteration)
    per_thread = max(1, int(target_mt_s / max(st_t, 1e-6) / len(iters)))
    mt_rows = cores * per_thread
    mt_t, mt_f = _oracle_sample(w, stat, counts, t, mt_rows, iters, cores)
    return {"value": mt_f / mt_t / 1e12, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
            "sample": _sample_text(w, mt_rows, iters, cores, mt_t),
            "single_thread": {"value": st_f / st_t / 1e12, "unit": "TFLOP/s", "cores": 1,
                              "sample": _sample_text(w, 1, iters[:1], 1, st_t)}}


def workload_desc(w, counts) -> str:
    """The workload as both arms name it in `config.workload`."""
    window = "" if w.window_pct == 100 else f", caching window {w.window_pct}%"
    return (f"{w.name}: N={w.N} ({w.grid[0]}x{w.grid[1]}x{w.grid[2]}), H={w.H}, D={w.D}, "
            f"budgets={list(w.budgets)}, counts={list(counts)}, T={w.T}, "
            f"iterations={list(w.iters)}{window}")


def run_reference(args, dist, rank, world):
    """The oracle as the reference arm: each step is a bounded sample of the
    workload (partition, then one of the schedule's distinct iterations in turn
    at full size, with one attention query row per host core), timed on the
    host cores."""
    if rank != 0:
        return
    w = workload_of(args)
    stat, counts = synth.stat_for(w)
    t = host_inputs(w)
    iters = representative_iters(w, counts)
    cores = host_cores()
    rows = cores
    # step k samples iteration iters[k mod len(iters)]
    for k in range(args.warmup):
        _oracle_sample(w, stat, counts, t, rows, [iters[k % len(iters)]], cores)
    tot_t, tot_f = 0.0, 0.0
    for k in range(args.steps):
        el, f = _oracle_sample(w, stat, counts, t, rows, [iters[k % len(iters)]], cores)
        tot_t += el
        tot_f += f
    value = tot_f / tot_t / 1e12
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot_t / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(w, counts)},
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                         "sample": "per step: " + _sample_text(w, rows, iters, cores,
                                                               tot_t / args.steps)
                         + " (one of these iterations per step, in turn)"},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def memory_sweep():
    """Gather / KV-scatter / cached-Euler bandwidth from L2-sized to multi-GB
    footprints.  Each rep is timed alone with CUDA events after an L2 flush;
    bytes are the algorithmic bytes of the call (see `algorithmic`)."""
    import paper_2605_06892_gb300 as hsa
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    peaks, src = load_peaks()
    g = torch.Generator(device="cpu").manual_seed(7)

    def timed(fn, reps=10):
        for _ in range(3):
            fn()
        ts = []
        for _ in range(reps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        return statistics.median(ts)

    def report(kind, shape, nbytes, ms):
        gbs = nbytes / (ms * 1e-3) / 1e9
        print(json.dumps({"sweep": kind, "shape": shape, "bytes": nbytes, "ms": ms, "gbs": gbs,
                          "frac_hbm": gbs / peaks["hbm_gbs"], "peak_source": src}), flush=True)

    row = 3072                                   # one Wan-1.3B token row, 12 x 128 bf16
    for n in (8192, 32768, 131072, 262144, 524288):
        N = 2 * n
        src_t = torch.empty((N, row // 2), dtype=torch.bfloat16, device=dev).normal_()
        idx = torch.randperm(N, generator=g)[:n].sort().values.to(torch.int32).to(dev)
        dst = torch.empty((n, row // 2), dtype=torch.bfloat16, device=dev)
        ms = timed(lambda: hsa.hsa_gather_active(src_t, idx, n, dst, stream))
        report("gather", f"{n} rows x {row} B", n * (2 * row + 4), ms)
        del src_t, dst
        kc = torch.empty((N, 12, 128), dtype=torch.bfloat16, device=dev).normal_()
        vc = torch.empty_like(kc).normal_()
        kf = torch.empty((n, 12, 128), dtype=torch.bfloat16, device=dev).normal_()
        vf = torch.empty_like(kf).normal_()
        ms = timed(lambda: hsa.hsa_kv_sync_scatter(kc, vc, kf, vf, idx, n, stream))
        report("kv_scatter", f"{n} rows x 2 x {row} B", n * (4 * row + 4), ms)
        if n in (32768, 262144):
            tab = torch.empty((N, 64, 2), device=dev).uniform_(-1, 1)
            ms = timed(lambda: hsa.hsa_kv_sync_scatter_rope(kc, vc, kf, vf, idx, n, tab, stream))
            # K, V read and written, idx, and the token's 512-byte table row
            report("kv_scatter_rope", f"{n} rows x 2 x {row} B", n * (4 * row + 4 + 512), ms)
            del tab
        del kc, vc, kf, vf
    for C in (16, 128):
        for N in (1 << 16, 1 << 20, 1 << 22, 1 << 24):
            if N * C * 4 > (1 << 31):
                continue
            n = N // 2
            x = torch.empty((N, C), device=dev).normal_()
            vh = torch.empty_like(x).normal_()
            vfr = torch.empty((n, C), device=dev).normal_()
            pos = torch.full((N,), -1, dtype=torch.int32)
            act = torch.randperm(N, generator=g)[:n].sort().values
            pos[act] = torch.arange(n, dtype=torch.int32)
            pos = pos.to(dev)
            ms = timed(lambda: hsa.hsa_cached_euler(x, vh, vfr, pos, -0.025, n, stream))
            nbytes = (N - n) * 12 * C + n * 16 * C + 4 * N
            report("cached_euler", f"N={N} C={C}, half active", nbytes, ms)
            del x, vh, vfr, pos
    for C in (16, 128):
        for N in (1 << 20, 1 << 22, 1 << 24):
            if N * C * 4 > (1 << 31):
                continue
            x = torch.empty((N, C), device=dev).normal_()
            vh = torch.empty_like(x).normal_()
            vfr = torch.empty_like(x).normal_()
            pos = torch.arange(N, dtype=torch.int32, device=dev)
            stat = torch.zeros(N, device=dev)
            ms = timed(lambda: hsa.hsa_cached_euler_l1rel(x, vh, vfr, pos, -0.025, stat,
                                                          1.0 / 9, N, stream))
            report("cached_euler_l1rel", f"N={N} C={C}, all active", N * (20 * C + 12), ms)
            del x, vh, vfr, pos, stat
    assert hsa.hsa_get_device_error(stream) == 0


def main():
    args = parse()
    if args.memory_sweep:
        memory_sweep()
        return
    if args.impl == "reference":
        dist, rank, world, _ = dist_setup("gloo")
        run_reference(args, dist, rank, world)
        return
    dist, rank, world, local_rank = dist_setup("nccl")
    run_hsa(args, dist, rank, world, local_rank)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
