#!/usr/bin/env python3
"""Benchmark: drafts/s of the single-pass cascaded drafter on one GB300 per rank.

One step = fe_draft_forward + fe_build_tree over one batch of the workload (the whole
hot path: fused-feature input FCs, N cascade layers, LM head with fused softmax/top-k,
Backbone Expansion tree). Default workload: the largest single-GPU drafter, shaped like
LLaMA-3.3-70B (d=8192, 64 query / 8 KV heads x 128, F=28672, V=128256, N=8, B=1, P=2048,
k=10, bf16 weights and caches; 16.5 GB streamed per draft). The same JSON line carries a
record of the batched-serving workload (LLaMA-3.1-8B shape, B=32, ragged prefixes in
[256, 4096] over a 16-token page pool) with its own rate, roofline, e2e and CPU baseline.
Inputs are seeded synthetic tensors; every step streams all weights (GBs, far above the
129 MB L2), so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--also NAME ...]
                  [--impl ours|reference]

Per-kernel times come from the GPU's own stamps inside the graph the step runs as
(fe_profile_graph): each launch's first-CTA start and last-warp exit, so per family the
time a launch adds to the step (its end minus the previous launch's end) sums to the step.

Multi-GPU (torchrun): replicas only. Every rank drafts its own batch with its own copy
of the drafter; there is no collective on the data path (a barrier brackets the timed
region and the slowest rank's time is reported), so the scaling is weak.
"""
from __future__ import annotations

import argparse
import json
import os
import platform
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

HBM_FALLBACK_GBS = 6800.0      # used only when MEASURED_PEAKS.json is absent
BF16_FALLBACK_TFLOPS = 1900.0  # burst
BF16_FALLBACK_SUSTAINED = 1700.0


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="l33_70b")
    ap.add_argument("--also", nargs="*", default=["b32_l31"],
                    help="further workloads measured in the same run, as sub-records of the JSON line")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--profile-steps", type=int, default=30,
                    help="graph replays with per-kernel GPU stamps for the per-kernel roofline")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="oracle sample budget per workload")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true", help="skip the verification / loss / commit timings")
    ap.add_argument("--set", action="append", default=[], metavar="KEY=VALUE",
                    help="override a workload field (e.g. n_layers=1) for profiling runs")
    return ap.parse_args(argv)


# DRAM traffic of the dominant kernel family from an ncu capture (dram__bytes_read.sum +
# dram__bytes_write.sum over the linear launches of a one-layer draft of the workload,
# scaled to the full draft by the launches' shapes), with the SHA-256 of the kernel
# sources it was taken on: a changed kernel reports traffic null.
TRAFFIC = {
    # ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum,gpu__time_duration.sum -k regex:linear_kernel
    #     -s 18 -c 6 on `bench.py --workload l33_70b --set n_layers=1 --also ...` (one draft's six linear
    # launches: W_fuse, W_in, W_qkv, W_o, W_gate/up, W_down; the eight-layer draft repeats the last four)
    "l33_70b": {"bytes_per_draft": (402804480 + 2994944) + (268569600 + 35072)
                + 8 * ((167912448 + 59136) + (134362112 + 127232) + (939734272 + 508160) + (470002176 + 48896)),
                "sources": ("fe_stream.cuh", "fe_linear.cu", "fe_common.cuh"), "src": "db0896d91ededd9f"},
    # the same metrics with -k regex:linear_mma_kernel -s 18 -c 6 on `bench.py --workload b32_l31 --set
    # n_layers=1 --also ...` (the tensor-core products of the six phases; the six-layer draft repeats
    # the last four)
    "b32_l31": {"bytes_per_draft": (102318080 + 2932992) + (68232192 + 13312)
                + 6 * ((50930432 + 0) + (34153216 + 0) + (235487488 + 1959424) + (119891456 + 462080)),
                "sources": ("fe_linear_mma.cu", "fe_tc.cuh", "fe_common.cuh"), "src": "ee529b04c166ea62"},
}


def kernel_source_hash(sources) -> str:
    import hashlib
    hsh = hashlib.sha256()
    for n in sources:
        with open(os.path.join(ROOT, "paper_2509_20416_gb300", "csrc", n), "rb") as f:
            hsh.update(f.read())
    return hsh.hexdigest()[:16]


def peaks():
    """(HBM GB/s, bf16 TFLOP/s burst, bf16 TFLOP/s sustained, 'measured' | 'fallback')."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return (float(j["hbm_gbs"]), float(j["bf16_tflops"]),
                float(j.get("bf16_tflops_sustained", j["bf16_tflops"])), "measured")
    return HBM_FALLBACK_GBS, BF16_FALLBACK_TFLOPS, BF16_FALLBACK_SUSTAINED, "fallback"


def cpu_model() -> str:
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                k = line.split(":", 1)[0].strip().lower()
                if k in ("model name", "cpu model"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.processor() or platform.machine()


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x: float, ws: int, device) -> float:
    """The largest of the ranks' values (the slowest rank's time); the value itself at
    one process."""
    if ws <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(ws: int, B: int, seconds_per_step: float) -> float:
    """Whole-job drafts/s: every replica drafts its own B sequences per step, and the job's
    step takes as long as its slowest rank."""
    return ws * B / seconds_per_step


def family_times(launches, n_replays: int) -> dict:
    """Per kernel family, from in_step_times() summed over n_replays graph replays: launches
    per draft, the time the family adds to the step and its summed spans (us per draft).
    A tensor-core phase's operand prep counts with its phase ('linear_prep' -> 'linear',
    'lm_prep' -> 'lm_head'); the main launches alone are counted."""
    fam = {}
    for kind, span, add in launches:
        key = {"linear_prep": "linear", "lm_prep": "lm_head"}.get(kind, kind)
        c = fam.setdefault(key, {"launches": 0, "added_us": 0.0, "span_us": 0.0})
        if kind == key:
            c["launches"] += 1
        c["added_us"] += add
        c["span_us"] += span
    out = {}
    for key, c in fam.items():
        out[key] = {"launches_per_draft": c["launches"] / n_replays, "us_per_draft": c["added_us"] / n_replays,
                    "span_us_per_draft": c["span_us"] / n_replays}
    return out


def roofline_block(kernels: dict, kbytes: dict, kflops: dict, ms_step: float, alg_bytes: int, alg_flops: int,
                   traffic, n_replays: int) -> dict:
    """The dominant kernel family's HBM roofline (algorithmic bytes per launch over the time a
    launch adds inside the graph-replayed step), the whole step's, and the tensor-pipe
    fractions (algorithmic flops over time, against the measured bf16 peaks)."""
    hbm, tf_burst, tf_sus, kind = peaks()
    top = max((k for k in kernels if k in kbytes), key=lambda x: kernels[x]["us_per_draft"])
    kt = kernels[top]
    launches = max(kt["launches_per_draft"], 1e-9)
    us_per_launch = kt["us_per_draft"] / launches
    bpl = kbytes[top] / launches
    achieved = bpl / (us_per_launch * 1e-6) / 1e9
    step_gbs = alg_bytes / (ms_step * 1e-3) / 1e9
    step_tflops = alg_flops / (ms_step * 1e-3) / 1e12
    per_gemm = {}
    for k, fl in kflops.items():
        if k in kernels and kernels[k]["us_per_draft"] > 0:
            t = fl / (kernels[k]["us_per_draft"] * 1e-6) / 1e12
            per_gemm[k] = {"tflops": t, "frac_burst": t / tf_burst, "frac_sustained": t / tf_sus}
    return {"bound": "hbm", "kernel": top, "achieved": achieved, "peak": hbm, "unit": "GB/s",
            "frac": achieved / hbm, "peak_kind": kind, "traffic": traffic,
            "algorithmic_bytes_per_launch": bpl, "us_per_launch": us_per_launch,
            "span_us_per_launch": kt["span_us_per_draft"] / launches, "launches_per_draft": launches,
            "timing": (f"GPU %globaltimer stamps of every launch inside the graph-replayed step "
                       f"(fe_profile_graph, {n_replays} replays); per launch the time it adds to the step "
                       f"(its end minus the previous launch's end)"),
            "step": {"achieved": step_gbs, "frac": step_gbs / hbm, "algorithmic_bytes": alg_bytes},
            "tensor": {"algorithmic_flops": alg_flops, "tflops": step_tflops, "peak_burst": tf_burst,
                       "peak_sustained": tf_sus, "frac_burst": step_tflops / tf_burst,
                       "frac_sustained": step_tflops / tf_sus, "peak_kind": kind, "per_gemm_family": per_gemm}}


def make_problem(name: str, overrides=()):
    from fe_synth import workloads as wl
    kw = {}
    for o in overrides:
        k, v = o.split("=", 1)
        kw[k] = type(wl.WORKLOADS[name][k])(v) if k in wl.WORKLOADS[name] else float(v)
    cfg = wl.make_config(name, **kw)
    W = wl.make_weights(cfg)
    I = wl.make_inputs(cfg)
    ks, vs = wl.make_caches(cfg)
    return cfg, W, I, ks, vs


def time_oracle(cfg, W, I, ks, vs, budget_s: float, max_runs: int | None = None):
    """The fp64 oracle as it stands, on the host cores, over a bounded sample of drafts
    (sequence b = run % B). Returns (drafts/s, runs, threads, seconds)."""
    import oracle
    orc = oracle.load()
    B = cfg["B"]
    runs, t0 = 0, time.perf_counter()
    while True:
        b = runs % B
        orc.draft_seq(cfg, W, I["feat"][b].contiguous(), int(I["next_tok"][b]), int(I["prefix_len"][b]),
                      [k[b].contiguous() for k in ks], [v[b].contiguous() for v in vs], cfg["max_seq"],
                      cfg["top_k"], cfg["temperature"], want_logits=False)
        runs += 1
        el = time.perf_counter() - t0
        if (max_runs and runs >= max_runs) or (not max_runs and el >= budget_s and runs >= 2):
            break
    return runs / el, runs, orc.max_threads(), el


def workload_config(cfg, wl) -> dict:
    return {"workload": cfg.get("name", "") + "".join(f" {o}" for o in cfg.get("overrides", [])),
            "shape": wl.describe(cfg), "B": cfg["B"], "N": cfg["n_layers"],
            "top_k": cfg["top_k"], "d": cfg["d"], "vocab": cfg["vocab"], "accum": "f32",
            "l2": "inputs larger than L2 (every step streams all weights, >129 MB)" if cfg["dtype"] == "bf16"
            else "L2-resident (no flush)"}


def run_reference(args, ws, rank):
    """The oracle, timed on this machine's host cores (the reference arm of this benchmark)."""
    if rank != 0:
        return
    from fe_synth import workloads as wl
    cfg, W, I, ks, vs = make_problem(args.workload, args.set)
    cfg["name"] = args.workload
    cfg["overrides"] = list(args.set)
    # warm-up runs, then a bounded number of timed steps (one draft of sequence step % B each)
    time_oracle(cfg, W, I, ks, vs, 0, max_runs=max(1, min(args.warmup, 2)))
    one, _, thr, _ = time_oracle(cfg, W, I, ks, vs, 0, max_runs=1)
    steps = max(1, min(args.steps, int(120.0 * one)))  # keep the arm within ~2 minutes
    rate, runs, thr, el = time_oracle(cfg, W, I, ks, vs, 0, max_runs=steps)
    value = rate  # drafts/s (one sequence's N-token draft per step)
    line = {"metric": "drafts/s", "value": value, "unit": "drafts/s", "n_gpus": ws, "steps": runs,
            "warmup": args.warmup, "ms_per_step": 1000.0 * el / runs, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded generator)",
            "config": workload_config(cfg, wl), "impl": "reference",
            "cpu_baseline": {"value": value, "unit": "drafts/s", "cores": thr, "kind": "oracle",
                             "cpu_model": cpu_model(),
                             "sample": f"{runs} single-sequence drafts of the workload"},
            "e2e": {"value": value, "unit": "drafts/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def measure(args, name: str, overrides, ws: int, rank: int, local: int, extras: bool) -> dict:
    """One workload: the timed steps, e2e, in-graph per-kernel times, roofline and (rank 0,
    one process) the oracle's rate. Returns the record (on every rank)."""
    import torch
    import paper_2509_20416_gb300 as fe
    from fe_synth import workloads as wl

    cfg, W, I, ks, vs = make_problem(name, overrides)
    cfg["name"] = name
    cfg["overrides"] = list(overrides)
    B, N, k = cfg["B"], cfg["n_layers"], cfg["top_k"]
    h = fe.fe_draft_init(dict(cfg, max_batch=B), W)
    if cfg["page_size"]:
        table, n_pages = wl.page_plan(cfg, I["prefix_len"])
        kd = [wl.paginate(cfg, t, table, n_pages).cuda() for t in ks]
        vd = [wl.paginate(cfg, t, table, n_pages).cuda() for t in vs]
        table = table.cuda()
    else:
        kd, vd, table, n_pages = [t.cuda() for t in ks], [t.cuda() for t in vs], None, 0
    feat, tok, plen = I["feat"].cuda(), I["next_tok"].cuda(), I["prefix_len"].cuda()
    out = fe.alloc_outputs(h, B, k)
    tree = fe.alloc_tree(h, B, k)
    stream = torch.cuda.current_stream()

    def step():
        fe.fe_draft_forward(h, feat, tok, plen, kd, vd, k, cfg["temperature"], page_table=table,
                            n_pages=n_pages, out=out, stream=stream)
        fe.fe_build_tree(h, tok, out["topk_id"], k, out=tree, stream=stream)

    def barrier():
        if ws > 1:
            import torch.distributed as dist
            dist.barrier()

    def check(where):
        st = fe.fe_last_device_status(h)
        if st != fe.FE_OK:
            raise SystemExit(f"{name}: device status {where}: {fe.fe_status_str(st)}")

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    check("after warm-up")

    sampler = ClockSampler(local)
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    e1.synchronize()
    torch.cuda.synchronize()
    barrier()
    clocks = sampler.stop()
    ms = max_over_ranks(e0.elapsed_time(e1), ws, "cuda")
    ms_step = ms / args.steps
    value = job_rate(ws, B, ms_step / 1e3)
    check("after the timed region")

    # ---- the same step with stochastic drafting at T = 1 (Sec. 2.2, "sample k candidates") --
    # (outside the headline: its cost next to the greedy step)
    def step_sampled():
        fe.fe_draft_forward(h, feat, tok, plen, kd, vd, k, 1.0, page_table=table, n_pages=n_pages, out=out,
                            stream=stream, sample=True, seed=0x5EED)
        fe.fe_build_tree(h, tok, out["topk_id"], k, out=tree, stream=stream)

    for _ in range(3):
        step_sampled()
    n_smp = max(3, args.steps // 4)
    barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(n_smp):
        step_sampled()
    e1.record(stream)
    e1.synchronize()
    ms_smp = max_over_ranks(e0.elapsed_time(e1), ws, "cuda") / n_smp
    smp_launches = []
    for _ in range(5):
        smp_launches.extend(fe.in_step_times(fe.fe_profile_graph(
            h, feat, tok, plen, kd, vd, k, 1.0, page_table=table, n_pages=n_pages, out=out, tree=tree,
            stream=stream, sample=True, seed=0x5EED)))
    smp_fam = family_times(smp_launches, 5)
    check("after the sampled steps")
    sampled = {"temperature": 1.0, "seed": 0x5EED, "steps": n_smp, "ms_per_step": ms_smp,
               "value": job_rate(ws, B, ms_smp / 1e3), "unit": "drafts/s",
               "lm_head_us_per_draft": smp_fam.get("lm_head", {}).get("us_per_draft"),
               "note": "the same step with sample=1 (Gumbel-top-k draws without replacement at T = 1); "
                       "lm_head_us_per_draft from GPU stamps inside the replayed graph"}

    # ---- end to end through the public API with host buffers ------------------------------
    # fe_draft_step_host: host inputs -> (pinned staging -> device copy, draft, tree, device
    # -> pinned copy, as one CUDA graph) -> host outputs; the call returns with the outputs
    # in host memory
    host_in = {n: t.contiguous().pin_memory() for n, t in (("feat", I["feat"]), ("tok", I["next_tok"]),
                                                           ("plen", I["prefix_len"]))}
    host_out = fe.alloc_host_step_outputs(h, B, k)
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out.values())

    def e2e_step():
        fe.fe_draft_step_host(h, host_in["feat"], host_in["tok"], host_in["plen"], kd, vd, k, cfg["temperature"],
                              page_table=table, n_pages=n_pages, out=host_out, stream=stream)

    for _ in range(3):
        e2e_step()
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.e2e_steps):
        e2e_step()
    e2e_s = max_over_ranks((time.perf_counter() - t0) / args.e2e_steps, ws, "cuda")

    # ---- per-kernel times inside the graph-replayed step (GPU stamps) ---------------------
    launches, n_rep, steps_us = [], max(1, args.profile_steps), []
    for _ in range(n_rep):
        stamps = fe.fe_profile_graph(h, feat, tok, plen, kd, vd, k, cfg["temperature"], page_table=table,
                                     n_pages=n_pages, out=out, tree=tree, stream=stream)
        its = fe.in_step_times(stamps)
        launches.extend(its)
        steps_us.append(sum(a for _, _, a in its))
    check("after the stamped replays")
    kernels = family_times(launches, n_rep)
    stamped_us = statistics.median(steps_us)

    # ---- verification / training / update calls (not part of the draft step) --------------
    extra = {}
    if extras:
        extra = time_extras(fe, h, cfg, wl, feat, tok, plen, kd, vd, table, n_pages, tree, stream, I, check)

    # ---- roofline of the dominant kernel family (and of the whole step) --------------------
    plist = I["prefix_len"].tolist()
    alg_bytes = wl.algorithmic_bytes(cfg, plist)
    alg_flops = wl.algorithmic_flops(cfg, plist)
    kbytes = wl.kernel_bytes(cfg, plist)
    kflops = wl.kernel_flops(cfg, plist)
    for kind, v in kernels.items():
        if kind in kbytes and v["us_per_draft"] > 0:
            v["algorithmic_bytes_per_draft"] = kbytes[kind]
            v["achieved_gbs"] = kbytes[kind] / (v["us_per_draft"] * 1e-6) / 1e9
        v["share_of_step"] = v["us_per_draft"] / (ms_step * 1e3)
    traffic = None
    tr = TRAFFIC.get(f"{name}{''.join(' ' + o for o in overrides)}")
    if tr and tr["src"] == kernel_source_hash(tr["sources"]) and "linear" in kernels:
        traffic = tr["bytes_per_draft"] / kernels["linear"]["launches_per_draft"]
    roof = roofline_block(kernels, kbytes, kflops, ms_step, alg_bytes, alg_flops, traffic, n_rep)
    if roof["kernel"] != "linear":
        roof["traffic"] = None
    launches_per_step = fe.fe_launch_count(h, B, True)

    rec = {"metric": "drafts/s", "value": value, "unit": "drafts/s", "n_gpus": ws, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": ms_step, "us_per_draft": ms_step * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": cfg["dtype"],
           "data": "synthetic (seeded generator)", "config": workload_config(cfg, wl),
           "roofline": roof, "kernels": kernels,
           "in_step": {"stamped_step_us": stamped_us, "families_sum_us": sum(v["us_per_draft"] for v in kernels.values()),
                       "event_step_us": ms_step * 1e3,
                       "note": "the per-family added times partition the stamped span of one graph replay "
                               "(first kernel start to tree kernel end), which lies inside the event-timed step"},
           "e2e": {"value": job_rate(ws, B, e2e_s), "unit": "drafts/s", "h2d_bytes_per_step": h2d,
                   "d2h_bytes_per_step": d2h,
                   "call": "fe_draft_step_host (host inputs and outputs; copies, draft and tree in one graph; "
                           "returns with the outputs in host memory)"},
           "gpu_launches": launches_per_step * args.steps, "launches_per_step": launches_per_step,
           "clocks": clocks, "sampled": sampled}
    rec.update(extra)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        rate, runs, thr, el = time_oracle(cfg, W, I, ks, vs, args.cpu_seconds)
        rec["cpu_baseline"] = {"value": rate, "unit": "drafts/s", "cores": thr, "kind": "oracle",
                               "cpu_model": cpu_model(),
                               "sample": f"{runs} single-sequence drafts of the workload ({el:.1f} s)"}
    h.close()
    del W, ks, vs, kd, vd
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return rec


def time_extras(fe, h, cfg, wl, feat, tok, plen, kd, vd, table, n_pages, tree, stream, I, check) -> dict:
    """fe_verify_greedy, fe_draft_loss and fe_commit on the same workload (outside the step)."""
    import torch
    B, N, k = cfg["B"], cfg["n_layers"], cfg["top_k"]
    T = 1 + N * k
    g = torch.Generator().manual_seed(1)
    target_next = torch.randint(0, cfg["vocab"], (B, T), generator=g, dtype=torch.int32).cuda()
    vout = fe.fe_verify_greedy(h, plen, tree, target_next, k, stream=stream)
    for _ in range(3):
        fe.fe_verify_greedy(h, plen, tree, target_next, k, out=vout, stream=stream)
    v0, v1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    v0.record(stream)
    for _ in range(100):
        fe.fe_verify_greedy(h, plen, tree, target_next, k, out=vout, stream=stream)
    v1.record(stream)
    v1.synchronize()
    verify_us = 1000.0 * v0.elapsed_time(v1) / 100

    V, d = cfg["vocab"], cfg["d"]
    # lossless verification of a sampled tree (fe_verify_sampled): a T = 1 sampled draft's tree,
    # draw ranks and q = softmax(logits), synthetic target distributions per node
    smp = fe.alloc_outputs(h, B, k)
    logits = torch.empty((B, N, V), device="cuda")
    fe.fe_draft_forward(h, feat, tok, plen, kd, vd, k, 1.0, page_table=table, n_pages=n_pages, out=smp,
                        dbg_logits=logits, stream=stream, sample=True, seed=0x5EED)
    stree = fe.fe_build_tree(h, tok, smp["topk_id"], k, stream=stream)
    q = torch.softmax(logits, dim=-1)
    nxt = torch.clamp(stree["depth"], max=N - 1).long()
    p = torch.softmax(logits[torch.arange(B, device="cuda")[:, None], nxt]
                      + 0.5 * torch.randn((B, T, V), generator=g).cuda(), dim=-1)
    u_acc = torch.rand((B, T), generator=g).clamp(1e-7, 1 - 1e-7).cuda()
    u_bonus = torch.rand((B, T), generator=g).clamp(1e-7, 1 - 1e-7).cuda()
    vs_out = fe.fe_verify_sampled(h, stree, smp["topk_rank"], q, p, u_acc, u_bonus, k, stream=stream)
    for _ in range(3):
        fe.fe_verify_sampled(h, stree, smp["topk_rank"], q, p, u_acc, u_bonus, k, out=vs_out, stream=stream)
    v0.record(stream)
    for _ in range(20):
        fe.fe_verify_sampled(h, stree, smp["topk_rank"], q, p, u_acc, u_bonus, k, out=vs_out, stream=stream)
    v1.record(stream)
    v1.synchronize()
    verify_sampled_us = 1000.0 * v0.elapsed_time(v1) / 20
    accepted = int(vs_out["n_accept"].sum())
    del p, q, logits
    check("after the sampled verification")

    teacher = torch.softmax(torch.randn((B, N, V), generator=g), dim=-1).cuda()
    target_feat = torch.randn((N, B, d), generator=g).cuda()
    for _ in range(3):
        fe.fe_draft_loss(h, feat, tok, plen, kd, vd, teacher, target_feat, k, page_table=table, n_pages=n_pages,
                         stream=stream)
    v0.record(stream)
    for _ in range(10):
        fe.fe_draft_loss(h, feat, tok, plen, kd, vd, teacher, target_feat, k, page_table=table, n_pages=n_pages,
                         stream=stream)
    v1.record(stream)
    v1.synchronize()
    loss_us = 1000.0 * v0.elapsed_time(v1) / 10
    check("after the loss forward")

    # fe_commit of N accepted rows per sequence, written over rows the caches already hold
    # (P_b - N ..), so paged pools need no new pages
    cfeat = torch.randn((B, N, 3 * d), generator=g).to(wl.torch_dtype(cfg)).cuda()
    ctok = torch.randint(0, cfg["vocab"], (B, N), generator=g, dtype=torch.int32).cuda()
    cn = torch.full((B,), N, dtype=torch.int32).cuda()
    cplen = torch.clamp(I["prefix_len"] - N, min=0).to(torch.int32).cuda()
    for _ in range(3):
        fe.fe_commit(h, cfeat, ctok, cn, cplen, kd, vd, page_table=table, n_pages=n_pages, stream=stream)
    v0.record(stream)
    for _ in range(5):
        fe.fe_commit(h, cfeat, ctok, cn, cplen, kd, vd, page_table=table, n_pages=n_pages, stream=stream)
    v1.record(stream)
    v1.synchronize()
    commit_us = 1000.0 * v0.elapsed_time(v1) / 5
    check("after the commits")
    return {"verify_greedy": {"us_per_call": verify_us, "sequences": B, "tree_nodes": T,
                              "note": "fe_verify_greedy after the step (positions + greedy acceptance walk)"},
            "verify_sampled": {"us_per_call": verify_sampled_us, "sequences": B, "tree_nodes": T,
                               "accepted_tokens": accepted,
                               "note": "fe_verify_sampled on a T = 1 sampled draft's tree (recursive rejection "
                                       "sampling in draw order, Sec. 2.4); synthetic target distributions"},
            "commit": {"us_per_call": commit_us, "rows_per_sequence": N,
                       "note": "fe_commit of N accepted rows per sequence (Sec. 2.4 Update and Iterate): "
                               "Eq. 1 and the cascade over the rows, one weight stream per 32 rows; "
                               "outside the timed step"},
            "draft_loss": {"us_per_call": loss_us,
                           "note": "fe_draft_loss: the draft with logits [B,N,V] and hidden states written out, "
                                   "then CE + Smooth L1 (Sec. 2.3); outside the timed step"}}


def main():
    args = parse()
    ws, rank, local = dist_env()
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return
    import torch
    torch.cuda.set_device(local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    line = measure(args, args.workload, args.set, ws, rank, local, extras=not args.no_extras)
    subs = {}
    for name in args.also or []:
        if name == args.workload:
            continue
        subs[name] = measure(args, name, (), ws, rank, local, extras=False)
    if subs:
        line["workloads"] = subs
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
