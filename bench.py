#!/usr/bin/env python3
"""Throughput of the GraphPO advantage path on GB300.

A step = one pass of the whole path (validation/planning, row statistics,
similarity merge, per-group scores and advantages, per-token scatter) over one
synthetic batch with the shape of the math RLVR workload (128 prompts x 16
rollouts, ~16 steps, lognormal lengths with a 2k-token median, bf16 d=1024
state embeddings); `--config` picks another shape.  Inputs are resident in HBM;
L2 is flushed (a 256 MiB write) before every timed step; every step is timed on
the device with CUDA events on the launching stream.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config math]

The same line carries `per_config`: the path timed the same way on each of the
other workload shapes (tiny, agentic search, wide groups, full batch, and the
branching-rollout tree layout), each with its own stage times, clocks and roofline.

Roofline: the bound of a kernel is the slower of its algorithmic bytes at the
measured HBM copy peak and its algorithmic FLOPs (the cosine GEMM's comparable upper
triangle) at the measured bf16 tensor peak.  The fp32 work of the compensated eta
statistics is an implementation device, not the method's work: it is reported apart
(`alu_note`), never as the bound.

Multi-GPU (torchrun, one rank per GPU): every rank runs its own batch of the same
shape (weak scaling, no collective on the data path); value = tokens of all ranks
divided by the slowest rank's time.  `--impl reference` times the CPU oracle.
Prints one JSON line on rank 0.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

L2_FLUSH_BYTES = 256 << 20
METRIC = "advantage-labelled rollout tokens/s & graphs/s; fraction of HBM roofline"
WORKLOADS = {
    "tiny": "tiny: 8 prompts x 8 rollouts x 6 steps, fp32 d=256, kappa 0.9",
    "math": "math RLVR shape: 128 prompts x 16 rollouts, ~16 steps, lognormal lengths (median 2k, cap 8k), "
            "bf16 d=1024, 32 centroids/prompt, sigma 0.08, rewards Bernoulli(Beta(2,2))",
    "agentic": "agentic-search shape: 256 prompts x 8 rollouts, 4-10 steps of 64-1024 tokens, bf16 d=1024, "
               "16 centroids/prompt, rewards Bernoulli(0.3)",
    "wide": "wide groups: 64 prompts x 64 rollouts x 32 steps (2048 states/group), bf16 d=2048, "
            "64 centroids/prompt, sigma 0.06",
    "full": "full batch: 512 prompts x 16 rollouts, ~20 steps, lognormal lengths (median 4k, cap 16k), "
            "bf16 d=1024, 48 centroids/prompt",
    "tree": "branching rollouts (tree layout): 128 prompts, branching schedule {2,5,4,2,2} (<= 292 states and "
            "160 leaves per prompt), edges of 64-512 tokens, bf16 d=1024, 32 centroids/prompt, sigma 0.08, "
            "rewards Bernoulli(Beta(2,2))",
}


def make_workload(name, seed_offset=0):
    from paper_2606_18954_gb300 import workloads as W
    if name in W.TREE_CONFIGS:
        return W.make_tree_batch(W.TREE_CONFIGS[name], seed=W.config_seed(name) + seed_offset)
    return W.make_batch(W.CONFIGS[name], seed=W.config_seed(name) + seed_offset)


def batch_tokens(b):
    return int(b["total_tokens"]) if b.get("parent") is not None else int(b["rollout_token_off"][-1])


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def alu_peak_tops():
    """fp32 CUDA-core issue peak in tera lane-operations/s: 152 SMs x 128 fp32 lanes x the
    measured maximum SM clock (2070 MHz on the GB300s)."""
    mhz = 2070.0
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mhz = float(json.load(f).get("sm_max_mhz", mhz))
    except Exception:
        pass
    return 152 * 128 * mhz * 1e6 / 1e12


def algorithmic(b):
    """Bytes and FLOPs of the path and of each stage (one launch each)."""
    import numpy as np
    N = len(b["step_len"])
    R = len(b["reward"])
    G = len(b["group_rollout_off"]) - 1
    T = batch_tokens(b)
    d = b["emb"].shape[1]
    esz = 2 if b["emb_dtype"] == "bf16" else 4
    zb = N * d * esz
    tree = b.get("parent") is not None
    if tree:
        ng = np.diff(b["group_state_off"]).astype(np.float64)
        meta = 4 * N + 16 * (G + 1)  # parents + group rollout / state / token offsets
    else:
        so, go = b["rollout_step_off"], b["group_rollout_off"]
        ng = (so[go[1:]] - so[go[:-1]]).astype(np.float64)
        meta = 12 * R
    flops = float(d * (ng ** 2).sum())  # comparable upper triangle: 2 d n^2 / 2 per group
    path_bytes = zb + 4 * N + meta + R + 4 * T
    # exact_stats: per embedding element two exact products (|z|^2 and the parent dot) and two
    # compensated additions (TwoSum: 6 operations plus the error accumulation): 16 fp32 operations
    alu_x = 16.0 * N * d
    stages = {
        "exact_stats": (zb + 16 * N, 0.0, alu_x),
        "tree_prep": (meta + 4 * N + R + 24 * N, 0.0),
        "prep": (4 * (G + 1) + 12 * (R + 1) + 4 * N + R + 8 * N + 4 * R, 0.0),
        "row_stats": (zb + 8 * N, 0.0),
        "similarity": (zb + 12 * N, flops),
        "groups": (8 * N + R + 12 * R + 4 * N + 17 * N + 8 * N, 0.0),
        "tokens": (4 * T + 8 * N + 4 * N + 4 * N, 0.0),
        # the group-resident kernels do the whole path, the compensated statistics included
        "fused": (path_bytes, flops, alu_x),
        "fused_f32": (path_bytes, flops, alu_x),
    }
    return dict(N=N, R=R, G=G, T=T, path_bytes=path_bytes, flops=flops, stages=stages)


class ClockSampler:
    """nvidia-smi clock and throttle-reason samples during the timed region."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id):
        self.index = None
        self.proc = None
        self.path = os.path.join("/tmp", f"gpo_clocks_{os.getpid()}.csv")
        try:
            lines = subprocess.run(["nvidia-smi", "--query-gpu=index,pci.bus_id", "--format=csv,noheader"],
                                   capture_output=True, text=True, timeout=20).stdout.splitlines()
            for ln in lines:
                idx, bid = [x.strip() for x in ln.split(",")]
                if bus_id and bid.lower().endswith(bus_id.lower()[-10:]):
                    self.index = idx
            if self.index is None and lines:
                self.index = lines[0].split(",")[0].strip()
        except Exception:
            pass

    def __enter__(self):
        try:
            cmd = ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.index is not None:
                cmd += ["-i", self.index]
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        try:
            rows = [[p.strip() for p in ln.split(",")] for ln in open(self.path) if ln.count(",") >= 7]
        except Exception:
            pass
        num = lambda x: float(x) if x.replace(".", "", 1).isdigit() else None
        sm = [v for v in (num(r[0]) for r in rows) if v is not None]
        mx = [v for v in (num(r[1]) for r in rows) if v is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[4:8]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "gpu_index": self.index}


def kernel_source_sha256(kernel_file):
    """Hash of a kernel's source file and the shared headers of the library."""
    csrc = os.path.join(ROOT, "paper_2606_18954_gb300", "csrc")
    h = hashlib.sha256()
    for name in [kernel_file] + sorted(f for f in os.listdir(csrc) if f.endswith(".cuh")):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def traffic_for(kernel_file, workload):
    """DRAM bytes per launch from the committed ncu summary of this kernel on this workload,
    if the kernel's sources are unchanged since the capture."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            t = json.load(f)
        ent = t[kernel_file][workload]
        if kernel_source_sha256(kernel_file) != ent["source_sha256"]:
            return None, "kernel changed since the capture"
        return float(ent["bytes_per_launch"]), ent.get("note", "")
    except Exception:
        return None, "no capture"


STAGE_SOURCE = {"prep": "gpo_prep.cu", "tree_prep": "gpo_prep.cu", "exact_stats": "gpo_prep.cu",
                "row_stats": "gpo_prep.cu", "similarity": "gpo_sim_tc.cu",
                "groups": "gpo_group.cu", "tokens": "gpo_prep.cu", "fused": "gpo_fused.cu",
                "fused_f32": "gpo_fused_f32.cu"}


def cpu_baseline(b, budget_s=6.0, max_groups=None):
    import numpy as np
    import oracle
    from paper_2606_18954_gb300 import workloads as W
    cores = len(os.sched_getaffinity(0))
    G = len(b["group_rollout_off"]) - 1
    sub, sample = b, f"the whole batch ({G} groups)"
    if max_groups is not None and G > max_groups:
        sub = W.sub_batch(b, range(max_groups))
        sample = f"the first {max_groups} of {G} groups"
    T = batch_tokens(sub)
    params = dict(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    oracle.run(W.sub_batch(sub, [0]), params, threads=1)  # build + warm
    times = []
    t_start = time.perf_counter()
    while True:
        t0 = time.perf_counter()
        oracle.run(sub, params, threads=cores, want={"adv"})
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start > budget_s and len(times) >= 2:
            break
    t = statistics.median(times)
    # the same oracle on one core, on the first groups of the sample (a few seconds)
    one = W.sub_batch(sub, range(min(8, len(sub["group_rollout_off"]) - 1)))
    t1 = []
    t_start = time.perf_counter()
    while True:
        t0 = time.perf_counter()
        oracle.run(one, params, threads=1, want={"adv"})
        t1.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start > budget_s / 3 and len(t1) >= 2:
            break
    return {"value": T / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{sample}, {len(times)} timed passes, median",
            "graphs_per_s": (len(sub["group_rollout_off"]) - 1) / t,
            "single_thread": {"value": batch_tokens(one) / statistics.median(t1), "unit": "tokens/s", "cores": 1,
                              "sample": f"the first {len(one['group_rollout_off']) - 1} groups, {len(t1)} passes, median"}}


def time_token_loss(P, gp, b, db, alg, flush, stream, args):
    """The policy loss (GraphPO Sec. 4.5 objective, dual form, edge normalisation, no KL term)
    on the batch's per-edge A_dual from the path and seeded log-probabilities, timed like the
    path (L2 flushed before every launch, CUDA events on the launching stream).  Algorithmic
    bytes per launch: log-probs, old log-probs and the gradient (12 bytes per token) plus
    every edge's first token, weight and advantage (16 bytes per edge)."""
    import torch
    from paper_2606_18954_gb300 import workloads as W
    T, N = alg["T"], alg["N"]
    nodes = gp.alloc_outputs(db, nodes=True)
    gp.compute_into(db, nodes, stream=stream)
    lp = W.make_logprobs(T, W.BASE_SEED + W.LOGP_SEED_OFFSET)
    logp = torch.from_numpy(lp["logp"]).to(db.step_len.device)
    old = torch.from_numpy(lp["old_logp"]).to(db.step_len.device)
    plan = gp.loss_plan(db, stream=stream)
    out = None
    for _ in range(args.warmup):
        out = gp.token_loss(db, plan, logp, old, edge_adv=nodes["edge_adv"], out=out, stream=stream)
    gp.check(stream)
    times = []
    for _ in range(args.steps):
        flush.zero_()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record(stream)
        gp.token_loss(db, plan, logp, old, edge_adv=nodes["edge_adv"], out=out, stream=stream)
        e.record(stream)
        e.synchronize()
        times.append(s.elapsed_time(e))
    gp.check(stream)
    ms = statistics.mean(times)
    res = {"ms": ms, "tokens_per_s": T / (ms / 1e3), "form": "dual", "norm": "edge", "beta_kl": 0.0,
           "loss": float(out["loss"].cpu()[0]), "launches_per_step": 1,
           "bytes": 12 * T + 16 * N}
    if not args.no_cpu_baseline:  # the loss oracle (numpy fp64) on the same batch and inputs
        import numpy as np
        from oracle import loss as OL
        A = np.random.default_rng(0).normal(0.0, 1.0, N)  # timing only: any per-edge advantages
        ts = []
        for _ in range(3):
            t0 = time.perf_counter()
            OL.token_loss(b, lp["logp"], lp["old_logp"], edge_adv=A)
            ts.append(time.perf_counter() - t0)
        res["cpu_baseline"] = {"value": T / statistics.median(ts), "unit": "tokens/s", "cores": 1, "kind": "oracle",
                               "sample": "the whole batch, 3 passes, median (numpy, one thread)"}
    return res


def time_efficiency(P, gp, db, out, wsp, flush, stream, args):
    """The path with and without its optional exploration-efficiency outputs (Eq. (eq1),
    both readings) and per-edge A_cor / A_eff / m_eff, timed like the path."""
    import torch

    def timed(o):
        for _ in range(args.warmup):
            gp.compute_into(db, o, workspace=wsp, stream=stream)
        ts = []
        for _ in range(args.steps):
            flush.zero_()
            s = torch.cuda.Event(enable_timing=True)
            e = torch.cuda.Event(enable_timing=True)
            s.record(stream)
            gp.compute_into(db, o, workspace=wsp, stream=stream)
            e.record(stream)
            e.synchronize()
            ts.append(s.elapsed_time(e))
        gp.check(stream)
        return statistics.mean(ts)

    extra = gp.alloc_outputs(db, edges=True, efficiency=True)
    with_eff = timed(extra)
    base = timed(out)
    return {"ms_with_outputs": with_eff, "ms_without": base, "overhead_ms": with_eff - base,
            "outputs": "group_eff, group_eff_graph, edge_cor, edge_eff, edge_eff_mask (and adv)"}


def time_layer_budget(P, b, flush, stream, args):
    """Per-layer graph construction (gpo_layer_budget: classes of the states sampled so far
    and next-layer budgets, GraphPO Sec. 4.2) after the second-to-last layer of a branching
    batch, timed like the path.  Algorithmic bytes per call: the embeddings of the states
    sampled so far, their parents and step lengths, the budgets out."""
    import torch
    from paper_2606_18954_gb300 import workloads as W
    H = len(b["spec"].schedule)
    t = W.truncate_tree(b, H - 1)
    db = P.Batch.from_arrays(t, device=stream.device)
    act = torch.as_tensor(t["active"], device=stream.device)
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    ws = gp.workspace(db)
    out = None
    for _ in range(args.warmup):
        out = gp.layer_budget(db, H - 1, b["spec"].schedule[H - 1], act, out=out, workspace=ws, stream=stream)
    gp.check(stream)
    times = []
    for _ in range(args.steps):
        flush.zero_()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record(stream)
        gp.layer_budget(db, H - 1, b["spec"].schedule[H - 1], act, out=out, workspace=ws, stream=stream)
        e.record(stream)
        e.synchronize()
        times.append(s.elapsed_time(e))
    gp.check(stream)
    N = len(t["step_len"])
    esz = 2 if t["emb_dtype"] == "bf16" else 4
    nbytes = N * t["emb"].shape[1] * esz + 4 * N + 4 * N + 4 * N + N
    ms = statistics.mean(times)
    res = {"ms": ms, "layer": H - 1, "states": N, "frontier": int((W.tree_depths(t) == H - 1).sum()),
           "active": int(t["active"].sum()), "states_per_s": N / (ms / 1e3), "bytes": nbytes,
           "b_next": int(b["spec"].schedule[H - 1])}
    if not args.no_cpu_baseline:  # the budget oracle on the first groups (a bounded sample)
        from oracle import budget as OB
        sub = W.truncate_tree(W.sub_batch(b, range(min(8, len(b["group_rollout_off"]) - 1))), H - 1)
        t0 = time.perf_counter()
        OB.layer_budget(sub, H - 1, int(b["spec"].schedule[H - 1]), sub["active"], dict(kappa=b["kappa"]))
        dt = time.perf_counter() - t0
        res["cpu_baseline"] = {"value": len(sub["step_len"]) / dt, "unit": "states/s", "cores": 1, "kind": "oracle",
                               "sample": f"the first {len(sub['group_state_off']) - 1} groups, one pass"}
    return res


def max_over_ranks(x, device=None):
    """The largest of the ranks' x (all ranks get it); x itself with one rank."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, device=None):
    """The sum of the ranks' x (all ranks get it); x itself with one rank."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def whole_job_value(tokens_all_ranks, ms_per_step):
    """Tokens/s of the whole job: every rank labels its own batch of the same shape (weak
    scaling); the job's tokens are all ranks' and it takes as long as its slowest rank."""
    return tokens_all_ranks / (ms_per_step / 1e3)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return ws, int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0"))


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2606_18954_gb300 import workloads as W
    import oracle
    b = make_workload(args.config)
    cores = len(os.sched_getaffinity(0))
    G = len(b["group_rollout_off"]) - 1
    max_groups = {"wide": 2, "full": 64}.get(args.config)
    sub, sample = b, f"the whole batch ({G} groups)"
    if max_groups and G > max_groups:
        sub = W.sub_batch(b, range(max_groups))
        sample = f"the first {max_groups} of {G} groups per step"
    T = batch_tokens(sub)
    params = dict(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    for _ in range(args.warmup):
        oracle.run(sub, params, threads=cores, want={"adv"})
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.run(sub, params, threads=cores, want={"adv"})
        times.append(time.perf_counter() - t0)
    ms = 1e3 * statistics.mean(times)
    value = T / (ms / 1e3)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOADS[args.config], "sample": sample},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "graphs_per_s": (len(sub["group_rollout_off"]) - 1) / (ms / 1e3)}
    print(json.dumps(line), flush=True)
    return 0


def kernel_roofline(name, stage_ms, alg, hbm, tc, workload):
    """Roofline of one kernel: its algorithmic bytes and FLOPs per launch (the method's
    work, as `algorithmic` counts it) over its average launch time; the bound is the
    slower of bytes at the HBM copy peak and FLOPs at the bf16 tensor peak (burst: each
    kernel runs alone, well under a millisecond)."""
    sb, sf = alg["stages"][name][:2]
    t = stage_ms[name] / 1e3
    if sf / (tc * 1e12) > sb / (hbm * 1e9):
        roof = {"bound": "tensor", "achieved": sf / t / 1e12, "peak": tc, "unit": "TFLOP/s",
                "algorithmic": sf, "peak_kind": "bf16 dense, burst"}
    else:
        roof = {"bound": "hbm", "achieved": sb / t / 1e9, "peak": hbm, "unit": "GB/s", "algorithmic": sb,
                "peak_kind": "HBM copy"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    traffic, tnote = traffic_for(STAGE_SOURCE.get(name, ""), workload)
    roof.update(kernel=name, ms_per_launch=stage_ms[name], traffic=traffic, traffic_note=tnote)
    return roof


def alu_note(name, stage_ms, alg):
    """The compensated statistics' fp32 operations of a kernel against the fp32 issue peak
    (an implementation device for the accuracy of eta, not part of the roofline)."""
    st = alg["stages"][name]
    if len(st) < 3 or not st[2]:
        return None
    peak = alu_peak_tops()
    achieved = st[2] / (stage_ms[name] / 1e3) / 1e12
    return {"kernel": name, "fp32_ops": st[2], "achieved": achieved, "peak": peak, "unit": "Top/s",
            "frac": achieved / peak, "peak_note": "152 SMs x 128 fp32 lanes x the max SM clock"}


def time_path(P, b, dev, stream, flush, args, barrier, bus):
    """The whole path on one batch: W warm-up steps, then K steps each timed on the device
    (CUDA events on the launching stream, L2 flushed before each), with the clocks sampled
    meanwhile; then K more steps with the library's per-kernel events."""
    import torch
    alg = algorithmic(b)
    db = P.Batch.from_arrays(b, device=dev)
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    out = gp.alloc_outputs(db)
    wsp = gp.workspace(db)
    for _ in range(args.warmup):
        gp.compute_into(db, out, workspace=wsp, stream=stream)
    gp.check(stream)
    torch.cuda.synchronize()
    # timed steps (the library's per-stage events are off here: they add a few microseconds)
    step_ms = []
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(bus) as clk:
        for _ in range(args.steps):
            flush.zero_()
            s = torch.cuda.Event(enable_timing=True)
            e = torch.cuda.Event(enable_timing=True)
            s.record(stream)
            gp.compute_into(db, out, workspace=wsp, stream=stream)
            e.record(stream)
            e.synchronize()
            step_ms.append(s.elapsed_time(e))
        torch.cuda.synchronize()
        barrier()
    gp.check(stream)
    # per-kernel durations: the same K steps again with CUDA events around each kernel
    stage_acc, nst = {}, 0
    gp.enable_timing(True)
    for _ in range(args.steps):
        flush.zero_()
        gp.compute_into(db, out, workspace=wsp, stream=stream)
        st = gp.stage_times()
        nst = len(st)
        for k, v in st.items():
            stage_acc[k] = stage_acc.get(k, 0.0) + v
    torch.cuda.synchronize()
    gp.check(stream)
    gp.enable_timing(False)
    return dict(alg=alg, db=db, gp=gp, out=out, wsp=wsp, step_ms=step_ms, clocks=clk.summary(),
                stage_ms={k: v / args.steps for k, v in stage_acc.items()}, launches_per_step=nst)


def config_summary(name, b, r, ms, tokens_all, n_ranks, peaks):
    """Throughput, stage times, clocks and rooflines of one shape."""
    hbm, tc = peaks[0], peaks[1]
    alg, stage_ms = r["alg"], r["stage_ms"]
    dom = max(stage_ms, key=stage_ms.get)
    path_t = max(alg["path_bytes"] / (hbm * 1e9), alg["flops"] / (tc * 1e12))
    res = {"workload": WORKLOADS[name], "ms_per_step": ms, "value": whole_job_value(tokens_all, ms),
           "unit": "tokens/s", "graphs_per_s": n_ranks * alg["G"] / (ms / 1e3),
           "groups": alg["G"], "rollouts": alg["R"], "states": alg["N"], "tokens": alg["T"],
           "d": int(b["emb"].shape[1]), "emb_dtype": b["emb_dtype"],
           "layout": "tree" if b.get("parent") is not None else "chain", "seed": _seed(name),
           "path_roofline": {"bytes": alg["path_bytes"], "flops": alg["flops"], "roofline_us": path_t * 1e6,
                             "bound": "tensor" if alg["flops"] / (tc * 1e12) > alg["path_bytes"] / (hbm * 1e9)
                             else "hbm", "frac": path_t / (ms / 1e3)},
           "stage_ms": stage_ms, "roofline": kernel_roofline(dom, stage_ms, alg, hbm, tc, name),
           "clocks": r["clocks"], "gpu_launches": r["launches_per_step"] * len(r["step_ms"])}
    note = alu_note(dom, stage_ms, alg)
    if note is not None:
        res["alu_note"] = note
    return res


def _seed(name):
    from paper_2606_18954_gb300 import workloads as W
    return W.config_seed(name)


def run_ours(args):
    import torch
    import paper_2606_18954_gb300 as P

    ws_n, rank, local = dist_env()
    if ws_n > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())
    P.build()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    peaks = load_peaks()
    hbm, tc, tc_sus, peak_src = peaks

    def barrier():
        if ws_n > 1:
            import torch.distributed as dist
            dist.barrier()

    bus = None
    try:
        bus = torch.cuda.get_device_properties(dev).pci_bus_id
    except Exception:
        pass

    b = make_workload(args.config, rank)
    r = time_path(P, b, dev, stream, flush, args, barrier, bus)
    alg, db, gp, out, wsp = r["alg"], r["db"], r["gp"], r["out"], r["wsp"]
    ms = max_over_ranks(sum(r["step_ms"]), dev) / args.steps
    tokens_all = sum_over_ranks(alg["T"], dev)  # the ranks' batches differ in their random lengths
    value = whole_job_value(tokens_all, ms)

    # end to end through the public API from pinned host buffers
    hb = P.Batch.from_arrays(b, device="cpu", pin=True)
    host_out = torch.empty(alg["T"], dtype=torch.float32, pin_memory=True)
    h2d = sum(t.numel() * t.element_size() for t in (hb.group_rollout_off, hb.rollout_step_off, hb.step_len,
                                                      hb.rollout_token_off, hb.emb, hb.reward, hb.parent,
                                                      hb.group_state_off, hb.group_token_off) if t is not None)
    for _ in range(max(1, args.warmup // 2)):
        gp.compute_host(hb, out=host_out)
    e2e_ms = []
    for _ in range(args.steps):
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record(stream)
        gp.compute_host(hb, out=host_out)
        e.record(stream)
        e.synchronize()
        e2e_ms.append(s.elapsed_time(e))
    e2e_t = max_over_ranks(statistics.mean(e2e_ms), dev)
    del hb, host_out

    loss = None if args.no_loss else time_token_loss(P, gp, b, db, alg, flush, stream, args)
    eff = None if args.no_loss else time_efficiency(P, gp, db, out, wsp, flush, stream, args)
    layer = None
    if not args.no_loss:  # per-layer merge on the branching workload (this one if branching)
        tb = b if b.get("parent") is not None else make_workload("tree", rank)
        layer = time_layer_budget(P, tb, flush, stream, args)
        layer["workload"] = WORKLOADS["tree"] if tb is not b else "this workload"

    head = config_summary(args.config, b, r, ms, tokens_all, ws_n, peaks)
    del r, db, gp, out, wsp

    # the other shapes, timed the same way (same K and W), one after another
    per_config = {}
    others = [c for c in (WORKLOADS if args.per_config == "all" else
                          ([] if args.per_config == "none" else args.per_config.split(",")))
              if c != args.config]
    for name in others:
        bo = make_workload(name, rank)
        ro = time_path(P, bo, dev, stream, flush, args, barrier, bus)
        mo = max_over_ranks(sum(ro["step_ms"]), dev) / args.steps
        to = sum_over_ranks(ro["alg"]["T"], dev)
        per_config[name] = config_summary(name, bo, ro, mo, to, ws_n, peaks)
        del ro, bo
        torch.cuda.empty_cache()

    if rank != 0:
        return 0
    roof = dict(head["roofline"])
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws_n, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": WORKLOADS[args.config], "groups": alg["G"], "rollouts": alg["R"],
                   "states": alg["N"], "tokens": alg["T"], "d": head["d"],
                   "emb_dtype": b["emb_dtype"], "layout": head["layout"],
                   "merge_rule": "noncausal", "kappa": b["kappa"], "w": b["w"],
                   "lambda_eff": b["lambda_eff"], "l2": "flushed by a 256 MiB write before every timed step",
                   "seed": _seed(args.config)},
        "graphs_per_s": head["graphs_per_s"],
        "path_roofline": head["path_roofline"],
        "stage_ms": head["stage_ms"],
        "roofline": roof,
        "e2e": {"value": whole_job_value(tokens_all, e2e_t), "unit": "tokens/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(4 * alg["T"]), "ms_per_step": e2e_t},
        "clocks": head["clocks"],
        "gpu_launches": head["gpu_launches"],
    }
    if "alu_note" in head:
        line["alu_note"] = head["alu_note"]
    if loss is not None:
        lb = loss.pop("bytes")
        achieved = lb / (loss["ms"] / 1e3) / 1e9
        traffic, tnote = traffic_for("gpo_loss.cu", args.config)
        loss["roofline"] = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                            "traffic": traffic, "traffic_note": tnote, "algorithmic_bytes": lb,
                            "peak_source": f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"}
        line["token_loss"] = loss
    if eff is not None:
        line["efficiency"] = eff
    if layer is not None:
        lb = layer.pop("bytes")
        achieved = lb / (layer["ms"] / 1e3) / 1e9
        layer["roofline"] = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                             "algorithmic_bytes": lb, "launches": "fused kernel alone (no row statistics)"}
        line["layer_budget"] = layer
    if per_config:
        line["per_config"] = per_config
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(b, max_groups={"wide": 2, "full": 64}.get(args.config))
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", choices=list(WORKLOADS), default="math")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--per-config", default="all",
                    help="other shapes timed into per_config: 'all', 'none' or a comma-separated list")
    ap.add_argument("--no-loss", action="store_true",
                    help="skip the measurements of the widenings (policy loss, efficiency outputs, per-layer merge)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
