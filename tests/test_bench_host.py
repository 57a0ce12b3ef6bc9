"""The benchmark's host-side arithmetic (CPU): algorithmic bytes and FLOPs per launch
as the roofline defines them (2d + 4 bytes per state, 13 per rollout, 4 per token,
d n_g^2 FLOPs per group; 16 fp32 operations per embedding element for the compensated
statistics), the fp32 issue peak, the measured-peak loader, the traffic lookup keyed
by the kernel's source hash, and the whole-job value."""
import json
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2606_18954_gb300 import workloads as W  # noqa: E402


def test_chain_algorithmic_work():
    b = W.make_batch(W.CONFIGS["math"].scaled(groups=3))
    a = bench.algorithmic(b)
    so, go = b["rollout_step_off"], b["group_rollout_off"]
    N, R, T, d = int(so[-1]), len(so) - 1, int(b["rollout_token_off"][-1]), 1024
    assert (a["N"], a["R"], a["G"], a["T"]) == (N, R, 3, T)
    assert a["path_bytes"] == N * (2 * d + 4) + 13 * R + 4 * T
    n_g = [int(so[go[g + 1]] - so[go[g]]) for g in range(3)]
    assert a["flops"] == float(d * sum(n * n for n in n_g))
    fused = a["stages"]["fused"]
    assert fused[0] == a["path_bytes"] and fused[1] == a["flops"] and fused[2] == 16.0 * N * d


def test_tree_algorithmic_work():
    spec = W.TREE_CONFIGS["tree"].scaled(groups=2, d=64)
    b = W.make_tree_batch(spec, seed=3)
    a = bench.algorithmic(b)
    N, R, G, T = len(b["parent"]), len(b["reward"]), 2, int(b["group_token_off"][-1])
    assert a["path_bytes"] == N * (2 * 64 + 4) + (4 * N + 16 * (G + 1)) + R + 4 * T
    assert a["flops"] == float(64 * sum(int(x) ** 2 for x in np.diff(b["group_state_off"])))


def test_fp32_issue_peak():
    """152 SMs x 128 fp32 lanes x the maximum SM clock (2070 MHz unless the measured file
    names another), in tera lane-operations per second."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    mhz = 2070.0
    if os.path.exists(path):
        mhz = float(json.load(open(path)).get("sm_max_mhz", mhz))
    assert bench.alu_peak_tops() == pytest.approx(152 * 128 * mhz * 1e-6, rel=1e-12)


def test_peaks_come_from_the_measured_file():
    hbm, bf16, bf16_sus, src = bench.load_peaks()
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        assert src == "measured" and hbm == float(p["hbm_gbs"]) and bf16 == float(p["bf16_tflops"])
    else:
        assert src == "fallback" and (hbm, bf16) == (6800.0, 1900.0)


def test_traffic_lookup_follows_the_kernel_source():
    t = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    for kernel, per in t.items():
        if kernel.startswith("_"):
            continue
        for workload, ent in per.items():
            got, note = bench.traffic_for(kernel, workload)
            if bench.kernel_source_sha256(kernel) == ent["source_sha256"]:
                assert got == float(ent["bytes_per_launch"])
            else:
                assert got is None and "changed" in note
    assert bench.traffic_for("gpo_fused.cu", "no such workload")[0] is None


def test_kernel_roofline_takes_the_slower_of_bytes_and_flops():
    """The bound of a kernel is max(bytes / HBM peak, FLOPs / tensor peak) of its
    algorithmic work; the fp32 work of the compensated statistics never decides it and
    is reported apart."""
    b = W.make_batch(W.CONFIGS["math"].scaled(groups=3))
    a = bench.algorithmic(b)
    hbm, tc = 6686.8, 1877.4
    ms = {"fused": 0.05, "exact_stats": 0.01, "similarity": 0.02}
    r = bench.kernel_roofline("fused", ms, a, hbm, tc, "math")
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(a["path_bytes"] / 0.05e-3 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / hbm)
    assert r["algorithmic"] == a["path_bytes"]
    # a contraction-heavy kernel: wide groups make the cosine GEMM the bound
    a2 = dict(a)
    a2["stages"] = dict(a["stages"], similarity=(1e6, 1e12))
    r2 = bench.kernel_roofline("similarity", ms, a2, hbm, tc, "wide")
    assert r2["bound"] == "tensor" and r2["achieved"] == pytest.approx(1e12 / 0.02e-3 / 1e12)
    # the statistics kernel has no FLOPs of the method: HBM-bound, its fp32 work in the note
    r3 = bench.kernel_roofline("exact_stats", ms, a, hbm, tc, "math")
    assert r3["bound"] == "hbm"
    note = bench.alu_note("exact_stats", ms, a)
    assert note["fp32_ops"] == a["stages"]["exact_stats"][2]
    assert note["frac"] == pytest.approx(note["achieved"] / bench.alu_peak_tops())
    assert bench.alu_note("similarity", ms, a) is None


def test_whole_job_value():
    assert bench.whole_job_value(4_000_000, 2.0) == pytest.approx(2e9)
