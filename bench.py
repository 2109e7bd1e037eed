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
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="hsa", choices=["hsa", "reference"])
    p.add_argument("--workload", default="wan13b", choices=list(synth.WORKLOADS))
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--memory-sweep", action="store_true",
                   help="HBM size sweep of gather, KV scatter and cached Euler (L2 flushed)")
    return p.parse_args()


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
            time.sleep(0.3)
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

class Layer:
    """Resident device state and inputs of one HSA layer workload."""

    def __init__(self, w: synth.Workload, dev, rep: int = 0):
        self.w, self.dev = w, dev
        N, H, D, C = w.N, w.H, w.D, w.C
        self.stat_h, self.counts = synth.stat_for(w, rep)
        seed = lambda t: synth.seed_for(w.cid, rep, t)  # noqa: E731
        dt = w.dtype
        self.stat = self.stat_h.to(dev)
        self.hidden = synth.normal((N, H * D), seed(1), dt).to(dev)
        self.q = synth.normal((N, H, D), seed(2), dt).to(dev)
        self.kc = synth.normal((N, H, D), seed(3), dt).to(dev)
        self.vc = synth.normal((N, H, D), seed(4), dt).to(dev)
        self.kf = synth.normal((N, H, D), seed(5), dt).to(dev)
        self.vf = synth.normal((N, H, D), seed(6), dt).to(dev)
        self.x = synth.normal((N, C), seed(7)).to(dev)
        self.vh = synth.normal((N, C), seed(8)).to(dev)
        self.v_fresh = synth.normal((N, C), seed(9)).to(dev)
        self.group_of = torch.empty(N, dtype=torch.int32, device=dev)
        self.idx = torch.empty(N, dtype=torch.int32, device=dev)
        self.pos = torch.empty(N, dtype=torch.int32, device=dev)
        self.gathered = torch.empty((N, H * D), dtype=self.hidden.dtype, device=dev)
        self.out = torch.empty((N, H, D), dtype=self.q.dtype, device=dev)
        self.iters = list(w.iters)

    def bytes_resident(self):
        return sum(t.numel() * t.element_size() for t in
                   (self.hidden, self.q, self.kc, self.vc, self.kf, self.vf, self.x, self.vh,
                    self.v_fresh, self.gathered, self.out))


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


# ---------------------------------------------------------------- hsa arm

def run_hsa(args, dist, rank, world, local_rank):
    import paper_2605_06892_gb300 as hsa
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    w = synth.WORKLOADS[args.workload]
    L = Layer(w, dev)
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

    def step(record):
        """One pass of the hot path; record(kind, fn) launches fn between events."""
        record("partition", lambda: hsa.hsa_partition(L.stat, T, budgets, L.counts, L.group_of,
                                                      ws, stream))
        for it in L.iters:
            n = n_of[it]
            ds = sig[it + 1] - sig[it]
            record("active", lambda: hsa.hsa_partition_active(L.group_of, T, budgets, it, L.idx,
                                                              L.pos, w.window_pct, stream))
            record("gather", lambda: hsa.hsa_gather_active(L.hidden, L.idx, n, L.gathered,
                                                           stream))
            record("scatter", lambda: hsa.hsa_kv_sync_scatter(L.kc, L.vc, L.kf, L.vf, L.idx, n,
                                                              stream))
            record("attention", lambda: hsa.hsa_active_attention(L.q, L.idx, n, L.kc, L.vc,
                                                                 L.out, 0.0, ws_att, stream))
            record("euler", lambda: hsa.hsa_cached_euler(L.x, L.vh, L.v_fresh, L.pos, ds, n,
                                                         stream))

    plain = lambda kind, fn: fn()  # noqa: E731
    for _ in range(args.warmup):
        flush.zero_()
        step(plain)
    torch.cuda.synchronize()
    assert hsa.hsa_get_device_error(stream) == 0

    per_kernel = {k: [] for k in kinds}
    step_events = []

    def timed(kind, fn):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        per_kernel[kind].append((a, b))

    barrier(dist)
    torch.cuda.synchronize()
    launches0 = hsa.hsa_launch_count()
    with ClockSampler(local_rank) as clocks:
        for _ in range(args.steps):
            flush.zero_()                       # L2 flush, outside the step's events
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s0.record(stream)
            step(timed)
            s1.record(stream)
            step_events.append((s0, s1))
        torch.cuda.synchronize()
    launches = hsa.hsa_launch_count() - launches0       # this library's kernels only
    barrier(dist)
    step_ms = [a.elapsed_time(b) for a, b in step_events]
    total_ms = max_over_ranks(dist, sum(step_ms), dev)
    ms_per_step = total_ms / args.steps
    kern_ms = {k: sum(a.elapsed_time(b) for a, b in v) / args.steps for k, v in per_kernel.items()}
    status = hsa.hsa_get_device_error(stream)
    assert status == 0, f"device error {status}"

    flops_step = sum(algorithmic(w, n_of[it])["attention_flops"] for it in L.iters)
    value = world * flops_step / (ms_per_step * 1e-3) / 1e12

    # memory-bound kernels: algorithmic bytes per step / time per step
    bytes_step = {k: sum(algorithmic(w, n_of[it])[k] for it in L.iters)
                  for k in ("gather", "scatter", "euler", "active")}
    peaks, peak_src = load_peaks()
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
            t = a.elapsed_time(b) / args.steps
            it_ms[e % n_it] += t
            if kind == "attention":
                att_ms[e % n_it] += t
    dense = dense_iteration(args, hsa, L, sig, flush, ws_att, stream)
    per_iter = {}
    for m, it in enumerate(L.iters):
        per_iter[str(it)] = {"n_active": n_of[it], "frac": n_of[it] / w.N, "ms": it_ms[m],
                             "attention_ms": att_ms[m], "vs_dense": it_ms[m] / dense["ms"]}
    dense_baseline = {
        "iteration_ms": dense["ms"], "attention_ms": dense["attention_ms"],
        "step_ms_all_dense": n_it * dense["ms"] + kern_ms["partition"],
        "step_vs_all_dense": ms_per_step / (n_it * dense["ms"] + kern_ms["partition"]),
        "what": f"{n_it} iterations with every token active (same kernels, |A| = N), "
                "against the measured step; L2 flushed before each dense iteration"}

    att_tflops = kernels["attention"]["tflops"]
    roofline = {"bound": "tensor", "achieved": att_tflops, "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "frac": att_tflops / peaks["bf16_tflops"],
                "traffic": profiled_traffic(w), "peak_source": f"{peak_src} bf16 burst",
                "frac_sustained": att_tflops / peaks["bf16_tflops_sustained"]}

    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) Q/K/V, lognormal statistic; no model weights)",
        "config": {"workload": workload_desc(w, L.counts),
                   "per_iteration": per_iter, "parallelism": f"replicas x{world}",
                   "l2": "flushed (256 MiB write) between steps; K/V cache and Q exceed L2",
                   "q_load": "index-driven (q_idx into the [N,H,D] query tensor)"},
        "kernels": kernels, "roofline": roofline, "dense_baseline": dense_baseline,
        "gpu_launches": launches,
        "clocks": clocks.summary(),
    }
    if not args.no_e2e:
        line["e2e"] = run_e2e(args, hsa, L, sig, n_of, stream, dev, dist, world, flops_step)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, L)
    if rank == 0:
        print(json.dumps(line), flush=True)


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


def run_e2e(args, hsa, L, sig, n_of, stream, dev, dist, world, flops_step):
    """Same step through the C ABI with host buffers (pinned).  Copies run on
    their own streams and overlap the kernels: each iteration's inputs are
    copied in two iterations ahead into a ring of three device buffers (so a
    large copy can overlap more than one short iteration), each attention
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

    def step():
        j0 = st["j"]
        loaded = {}
        with torch.cuda.stream(s_in):
            if st["stat_free"] is not None:
                s_in.wait_event(st["stat_free"])
            L.stat.copy_(h_stat, non_blocking=True)
            stat_ready = ev()
            stat_ready.record(s_in)

        def load(k):
            j = j0 + k
            b, n = bufs[j % nbuf], n_of[iters[k]]
            with torch.cuda.stream(s_in):
                if st["in_free"][j % nbuf] is not None:
                    s_in.wait_event(st["in_free"][j % nbuf])
                b["q"][:n].copy_(h_q[:n], non_blocking=True)
                b["kf"][:n].copy_(h_kf[:n], non_blocking=True)
                b["vf"][:n].copy_(h_vf[:n], non_blocking=True)
                b["vfr"][:n].copy_(h_vfr[:n], non_blocking=True)
                e = ev()
                e.record(s_in)
                loaded[k] = e

        for k in range(ahead):
            load(k)
        stream.wait_event(stat_ready)
        hsa.hsa_partition(L.stat, T, budgets, L.counts, L.group_of, ws, stream)
        st["stat_free"] = ev()
        st["stat_free"].record(stream)
        for k, it in enumerate(iters):
            if k + ahead < len(iters):
                load(k + ahead)
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

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    barrier(dist)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s_in)
    stream.wait_event(a)
    s_out.wait_event(a)
    for _ in range(args.steps):
        step()
    s_out.wait_stream(stream)
    s_out.wait_stream(s_in)
    b.record(s_out)
    torch.cuda.synchronize()
    barrier(dist)
    ms = max_over_ranks(dist, a.elapsed_time(b), dev) / args.steps
    assert hsa.hsa_get_device_error(stream) == 0
    return {"value": world * flops_step / (ms * 1e-3) / 1e12, "unit": "TFLOP/s",
            "ms_per_step": ms, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "copies": "pinned host buffers; inputs copied two iterations ahead on a copy "
                      "stream, outputs copied back on another, overlapping the kernels"}


def code_digest(text: str) -> str:
    """Digest of a CUDA source with its comments and whitespace removed, so
    that an edit to comments alone does not invalidate a profile."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    text = " ".join(text.split())
    return hashlib.sha256(text.encode()).hexdigest()[:16]


def profiled_traffic(w):
    """DRAM bytes per attention launch from the committed ncu summary, if it
    was taken on the current attention code (comments aside); else None."""
    path = os.path.join(ROOT, "profiles", f"attention_{w.name}.md")
    src = os.path.join(ROOT, "paper_2605_06892_gb300", "csrc", "hsa_attention.cu")
    try:
        digest = code_digest(open(src).read())
        fields = {}
        for line in open(path):
            if line.startswith("traffic_per_launch_bytes:") or line.startswith("code_sha256:"):
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
        if fields.get("code_sha256") == digest:
            return float(fields["traffic_per_launch_bytes"])
    except (OSError, KeyError, ValueError):
        pass
    return None


# ----------------------------------------------------------- CPU oracle leg

def _oracle_sample(w, stat, counts, tensors, rows_per_iter, iters):
    """The oracle's pass over one bounded sample of the workload: partition,
    active set, gather, scatter and cached Euler at full size, attention for
    `rows_per_iter` active query rows (all heads, all N keys) per iteration.
    Returns (seconds, attention FLOPs done)."""
    import oracle
    hidden, q, kc, vc, kf, vf, x, vh, vfr = tensors
    sig = oracle.sigmas(w.T, w.shift)
    t0 = time.perf_counter()
    g = oracle.partition(stat, w.T, w.budgets, counts)
    flops = 0.0
    for it in iters:
        idx, pos = oracle.active_set(g, w.T, w.budgets, it, w.window_pct)
        n = idx.numel()
        oracle.gather(hidden, idx)
        oracle.kv_scatter(kc, vc, kf[:n], vf[:n], idx)
        rows = idx[:rows_per_iter]
        oracle.attention(q, kc, vc, q_idx=rows)
        flops += 4.0 * rows.numel() * w.N * w.D * w.H
        oracle.cached_euler_f32(x, vh, vfr[:n], pos, float(sig[it + 1] - sig[it]))
    return time.perf_counter() - t0, flops


def _host_tensors(w, rep=0):
    seed = lambda t: synth.seed_for(w.cid, rep, t)  # noqa: E731
    dt = w.dtype
    N, H, D, C = w.N, w.H, w.D, w.C
    return (synth.normal((N, H * D), seed(1), dt), synth.normal((N, H, D), seed(2), dt),
            synth.normal((N, H, D), seed(3), dt), synth.normal((N, H, D), seed(4), dt),
            synth.normal((N, H, D), seed(5), dt), synth.normal((N, H, D), seed(6), dt),
            synth.normal((N, C), seed(7)), synth.normal((N, C), seed(8)),
            synth.normal((N, C), seed(9)))


def cpu_baseline(w, L=None, target_s=15.0):
    """Oracle timed on the host cores on a bounded sample (single thread)."""
    stat, counts = synth.stat_for(w)
    tensors = _host_tensors(w)
    t1, f1 = _oracle_sample(w, stat, counts, tensors, 1, w.iters[:1])
    per_row = t1 / max(f1, 1.0)
    rows = max(1, int(target_s / max(per_row * 4.0 * w.N * w.D * w.H, 1e-9) / len(w.iters)))
    t, f = _oracle_sample(w, stat, counts, tensors, rows, w.iters)
    return {"value": f / t / 1e12, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
            "sample": f"partition, active sets, gather, KV scatter and cached Euler at full "
                      f"size plus attention of {rows} active query rows x {w.H} heads x "
                      f"{w.N} keys in each of iterations {list(w.iters)}, fp64, "
                      f"{t:.1f} s single-threaded"}


def workload_desc(w, counts) -> str:
    """The workload as both arms name it in `config.workload`."""
    return (f"{w.name}: N={w.N} ({w.grid[0]}x{w.grid[1]}x{w.grid[2]}), H={w.H}, D={w.D}, "
            f"budgets={list(w.budgets)}, counts={list(counts)}, T={w.T}, "
            f"iterations={list(w.iters)}")


def run_reference(args, dist, rank, world):
    """The oracle as the reference arm: each step is a bounded sample of the
    workload (4 query rows per iteration), timed on the host cores."""
    if rank != 0:
        return
    w = synth.WORKLOADS[args.workload]
    stat, counts = synth.stat_for(w)
    tensors = _host_tensors(w)
    rows = 4
    for _ in range(args.warmup):
        _oracle_sample(w, stat, counts, tensors, rows, w.iters)
    tot_t, tot_f = 0.0, 0.0
    for _ in range(args.steps):
        t, f = _oracle_sample(w, stat, counts, tensors, rows, w.iters)
        tot_t += t
        tot_f += f
    value = tot_f / tot_t / 1e12
    sample = (f"oracle pass per step: full-size partition/active set/gather/scatter/Euler and "
              f"attention of {rows} query rows x {w.H} heads per iteration {list(w.iters)}")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot_t / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(w, counts)},
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
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
