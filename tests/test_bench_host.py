"""Host-side pieces of the benchmark, with no GPU: the workload names both arms
print, the summary of an extra workload run, and the DRAM traffic that the
roofline reports, read from the committed ncu summary of the attention kernel."""
import dataclasses
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import oracle  # noqa: E402
import synth  # noqa: E402


def test_workload_desc_names_the_window():
    w = synth.WORKLOADS["wan14b_720p"]
    _, counts = synth.stat_for(w)
    plain = bench.workload_desc(w, counts)
    assert plain.startswith("wan14b_720p: N=75600") and "window" not in plain
    w80 = dataclasses.replace(w, name="wan14b_720p_window80", window_pct=80)
    assert bench.workload_desc(w80, counts).endswith(", caching window 80%")


def test_also_summary_figures():
    w = synth.WORKLOADS["wan13b"]
    res = {
        "flops_step": 11.5e12, "ms_per_step": 6.0,
        "kernels": {"attention": {"tflops": 1900.0},
                    "gather": {"frac_hbm": 0.75}, "scatter": {"frac_hbm": 0.84},
                    "euler": {"frac_hbm": 0.2}, "partition": {"ms": 0.01}},
        "iterations": {"1": {"vs_dense": 1.0}, "0.5": {"vs_dense": 0.5}},
        "dense_baseline": {"step_vs_all_dense": 0.58, "ideal_vs_all_dense": 0.5833},
        "timing": {"graph_ms_per_step": 5.9}, "launches": 22, "clocks": {"sm_mhz": 2070.0}}
    peaks = {"bf16_tflops": 1897.5}
    out = bench.also_summary(w, (8190, 8190, 16380), 10, res, peaks, world=2)
    assert out["value"] == pytest.approx(2 * 11.5e12 / 6e-3 / 1e12)
    assert out["attention_frac_burst"] == pytest.approx(1900.0 / 1897.5)
    assert out["iterations_vs_dense"] == {"1": 1.0, "0.5": 0.5}
    assert out["step_vs_all_dense"] == 0.58 and out["ideal_vs_all_dense"] == 0.5833
    assert out["steps"] == 10 and out["gpu_launches"] == 22


def test_attention_traffic_profile_is_current():
    """The 720p layer's traffic summary carries the digest of the attention
    source it was measured on; the roofline uses it only while that digest
    matches the source (comments and whitespace aside).  The committed summary
    must match the committed kernel, and its bytes must lie between the
    algorithmic bytes and twice them."""
    w = synth.WORKLOADS["wan14b_720p"]
    _, counts = synth.stat_for(w)
    n_of = {it: oracle.active_count(w.budgets, counts, w.T, it, w.window_pct)
            for it in w.iters}
    got = bench.profiled_traffic(w, n_of)
    assert got is not None, "profiles/attention_wan14b_720p.md is stale for hsa_attention.cu"
    algo = sum(bench.algorithmic(w, n)["attention_bytes"] for n in n_of.values()) / len(n_of)
    assert algo < got < 2 * algo
