"""Benchmark: candidate plans evaluated per second on the burst-arrival window
(64 sessions, N=2000 activations, D=8 devices, M=8 models, P=16,384 plans per
GPU), plus the evaluation kernel's achieved HBM bandwidth against the measured
copy peak.

One step = the whole hot path over one batch: readiness forecast, evaluation
of every plan, top-k.  Inputs are resident in HBM before the timed region; L2
is flushed (a 256 MiB write, read back) between timed steps, which are timed one by one
with CUDA events on the library's stream.  ``e2e`` repeats the step through
wf_eval_topk_host, the C-ABI call that takes the plans in (page-locked) host
memory and returns the top-k and the forecast there; its host-to-device copy
(into one of two staging slots, overlapping the previous step's evaluation)
and the read-back lie inside the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gpu|reference]

Under torchrun every rank evaluates its own batch (plan indices offset by
rank * P; weak scaling) and rank 0 prints one JSON line.  ``--impl reference``
times the CPU oracle on the host cores on a bounded sample of the same batch.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "burst"
METRIC = "candidate plans evaluated/sec (N=2000,D=8)"
L2_FLUSH_BYTES = 256 << 20


def algorithmic_bytes_per_plan(N: int) -> int:
    """Compulsory traffic of one plan: place (N B) + order (2N B) + fusion and
    prefetch bits (2 ceil(N/8) B) read, makespan / p95 / GPU time (3 x 8 B) and
    status (4 B) written."""
    return N + 2 * N + 2 * ((N + 7) // 8) + 28


def host_cpu() -> dict:
    """The host the oracle runs on: logical cores and the CPU model as lscpu
    (or /proc/cpuinfo) names it."""
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() == "Model name":
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if model is None:
        try:
            with open("/proc/cpuinfo") as f:
                for line in f:
                    if line.lower().startswith("model name"):
                        model = line.split(":", 1)[1].strip()
                        break
        except OSError:
            pass
    import platform
    return {"nproc": os.cpu_count(), "cpu_model": model or platform.machine()}


def topk_launches(P: int, k: int) -> int:
    """Kernel launches of one wf_topk call: one CTA does select, compact and
    sort up to 16,384 plans; beyond, three kernels (tile bounds, compaction,
    final select and sort; the two scratch words are reset by memsets)."""
    return 1 if P <= 16384 else 3


def kernel_code(files: dict) -> str:
    """The evaluation kernels' code from the sources {name: text}: wf_eval.cu
    and wf_sweep.cu whole, and of wf_internal.cuh the device problem record
    and the #defines (the rest of that header is host-side: the context
    record and the launchers' declarations); comments, indentation and blank
    lines removed.  (No string literal in these files holds a comment marker.)"""
    import re
    hdr = files["wf_internal.cuh"]
    rec = re.search(r"struct wf_dev_problem \{.*?\n\};", hdr, flags=re.S)
    parts = [files["wf_eval.cu"], files["wf_sweep.cu"], rec.group(0) if rec else hdr,
             "\n".join(ln for ln in hdr.splitlines() if ln.startswith("#define"))]
    out = []
    for src in parts:
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        out += [ln for ln in (re.sub(r"//.*$", "", ln).strip() for ln in src.splitlines()) if ln]
    return "\n".join(out)


def kernel_source_hash() -> str:
    """sha256 (first 16 hex digits) of kernel_code(): an edit to a comment or
    to host-side declarations keeps the recorded counters, any edit to the
    kernels' code drops them."""
    files = {}
    for f in ("wf_eval.cu", "wf_sweep.cu", "wf_internal.cuh"):
        with open(os.path.join(ROOT, "paper_2609_03335_gb300", "csrc", f), encoding="utf-8") as fh:
            files[f] = fh.read()
    return hashlib.sha256(kernel_code(files).encode()).hexdigest()[:16]


def flush_l2(buf):
    """Flush L2 before a timed step: write the 256 MiB buffer (larger than
    L2), then read it back, so the write-backs of its dirty lines happen here
    and the step starts with a cold L2 of clean lines (none of its inputs)."""
    buf.zero_()
    buf.amax()


def read_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


def read_traffic(workload: str):
    """DRAM bytes per launch of the evaluation kernel from the committed ncu
    summary, only if it was taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", "eval_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except OSError:
        return None, None
    if d.get("kernel_hash") != kernel_source_hash() or workload not in d.get("per_launch", {}):
        return None, d.get("kernel_hash")
    return d["per_launch"][workload], d.get("kernel_hash")


def read_instructions(workload: str):
    """Warp instructions of one evaluation call from the same ncu summary (same
    kernel-source condition as the traffic)."""
    try:
        with open(os.path.join(ROOT, "profiles", "eval_traffic.json")) as f:
            d = json.load(f)
    except OSError:
        return None
    if d.get("kernel_hash") != kernel_source_hash():
        return None
    return d.get("warp_instructions", {}).get(workload)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 50 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = os.path.join("/tmp", f"wf_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        load = [s for s in sm if s > 0.5 * max(sm)] or sm
        return {"sm_mhz": float(np.median(load)), "sm_max_mhz": float(max(smax)),
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if os.environ.get("WF_BENCH_BACKEND", "nccl") == "nccl" else "gloo"
        dist.init_process_group(backend=backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if dist.get_backend() == "nccl" else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def run_reference(args, rank, world):
    """The CPU oracle, as it stands, timed on the host cores."""
    import oracle
    import wfgen
    if rank != 0:
        return
    w = wfgen.config(WORKLOAD)
    sample = 1024
    plans = wfgen.make_plans(w.problem, sample, w.plan_seed)
    oracle.build()
    for _ in range(args.warmup):
        oracle.eval_plans(w.problem, plans, 0, 64)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.eval_plans(w.problem, plans)
    dt = (time.perf_counter() - t0) / args.steps
    value = sample / dt
    line = {
        "impl": "reference", "metric": metric_of(w.problem), "value": value, "unit": "plans/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
        "data": "synthetic",
        "config": {"workload": f"{WORKLOAD}: {w.description}; oracle step = first {sample} plans of the batch",
                   "P": sample, "N": w.problem.N},
        "cpu_baseline": {"value": value, "unit": "plans/s", "cores": 1, "kind": "oracle",
                         "sample": f"first {sample} plans of the {WORKLOAD} batch per step, one thread",
                         **host_cpu()},
        "e2e": {"value": value, "unit": "plans/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def local_search_timing(wf, ctx, dp, prob, P, stream, flush, peak_gbs, k=32, rounds=3):
    """Local search around the batch's first k plans: P - k children per
    round (mutate -> evaluate -> merge; the context holds P plans).  The
    mutation kernel alone is timed too; it writes the child rows and reads
    the k parent rows (once from DRAM, then from L2)."""
    import torch
    N = prob.N
    P = P - k
    elite = wf.DevicePlans(dp.place[:k], dp.order[:k], dp.fuse[:k], dp.prefetch[:k], None, plan_base=0)
    er = wf.Results(k, dp.place.device)
    kids = wf.DevicePlans.empty(P, N, device=dp.place.device, plan_base=k)
    kr = wf.Results(P, dp.place.device)
    with torch.cuda.stream(stream):
        wf.wf_eval_plans(ctx, elite, er, stream)
        wf.wf_local_search(ctx, elite, er, kids, kr, seed=7, round0=0, rounds=1, n_ops=3, stream=stream)
        e = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        mut = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(5)]
        for r, (a, b) in enumerate(mut):
            flush_l2(flush)
            a.record(stream)
            wf.wf_mutate_plans(ctx, elite, kids, seed=7, round_=1 + r, n_ops=3, stream=stream)
            b.record(stream)
        flush_l2(flush)
        e[2].record(stream)
        wf.wf_local_search(ctx, elite, er, kids, kr, seed=7, round0=2, rounds=rounds, n_ops=3, stream=stream)
        e[3].record(stream)
    torch.cuda.synchronize()
    mut_ms = float(np.median([a.elapsed_time(b) for a, b in mut]))
    ls_ms = e[2].elapsed_time(e[3])
    # Compulsory DRAM bytes: every child row written once, the k parent rows
    # read once (the children's further reads of them hit L2).
    row = N + 2 * N + 2 * 4 * ((N + 31) // 32)
    bytes_per_child = row * (P + k) / P
    gbs = bytes_per_child * P / (mut_ms * 1e-3) / 1e9
    return {"k": k, "children_per_round": P, "rounds": rounds, "n_ops": 3,
            "ms_per_round": ls_ms / rounds, "children_per_s": P * rounds / (ls_ms * 1e-3),
            "mutate_kernel": {"ms": mut_ms, "timing": "median of 5 launches, L2 flushed before each", "bytes_per_child": bytes_per_child, "achieved_gbs": gbs,
                              "frac": gbs / peak_gbs if peak_gbs else None, "bound": "hbm"}}


def construct_timing(wf, ctx, prob, P, k, stream, flush, random_best, jitter=200000):
    """The plan constructor over a batch of P plans (jittered list schedules),
    timed on the device, then evaluated: its best makespan against the best
    of the random batch."""
    import torch
    dev = torch.device("cuda", torch.cuda.current_device())
    out = wf.DevicePlans.empty(P, prob.N, device=dev)
    res = wf.Results(P, dev)
    ids = torch.empty(k, dtype=torch.int32, device=dev)
    keys = torch.empty((k, 3), dtype=torch.int64, device=dev)
    e = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    with torch.cuda.stream(stream):
        wf.wf_construct_plans(ctx, out, seed=11, jitter_us=jitter, stream=stream)  # first call allocates
        flush_l2(flush)
        e[0].record(stream)
        wf.wf_construct_plans(ctx, out, seed=12, jitter_us=jitter, stream=stream)
        e[1].record(stream)
        wf.wf_eval_plans(ctx, out, res, stream)
        wf.wf_topk(ctx, res, P, k, ids, keys, stream)
    torch.cuda.synchronize()
    ms = e[0].elapsed_time(e[1])
    return {"plans": P, "jitter_us": jitter, "ms": ms, "plans_per_s": P / (ms * 1e-3),
            "best_makespan_us": int(keys[0, 0].item()), "random_batch_best_makespan_us": random_best}


def metric_of(prob):
    """The headline metric for the burst workload; the same form for others."""
    if WORKLOAD == "burst":
        return METRIC
    return f"candidate plans evaluated/sec (N={prob.N},D={prob.D}" + (f",S={prob.S})" if prob.S else ")")


def run_step(wf, ctx, dp, res, rel, comp, ids, keys, P, k, stream, side, ev=None):
    """One forecast / eval / top-k step.  The readiness forecast depends on the
    window only, not on the plans, so it runs on a second stream beside the
    evaluation, forked from and joined back into the step's stream with
    events; the step ends when both have.  ev: timing events (start, eval
    start, eval end, end, forecast start, forecast end) or None."""
    import torch
    fork = ev[0] if ev else torch.cuda.Event()
    fork.record(stream)
    side.wait_event(fork)
    if ev:
        ev[4].record(side)
    wf.wf_forecast_readiness(ctx, rel, comp, side)
    done = ev[5] if ev else torch.cuda.Event()
    done.record(side)
    if ev:
        ev[1].record(stream)
    wf.wf_eval_plans(ctx, dp, res, stream)
    if ev:
        ev[2].record(stream)
    wf.wf_topk(ctx, res, P, k, ids, keys, stream)
    stream.wait_event(done)
    if ev:
        ev[3].record(stream)


def issue_roofline(eval_ms, clk, sms, workload=None):
    """The integer-issue roofline of the evaluation call: its warp
    instructions (ncu, same kernel source) over its CUDA-event time, against
    4 warp instructions per clock per SM at the median SM clock sampled
    during the run."""
    inst = read_instructions(workload or WORKLOAD)
    mhz = (clk or {}).get("sm_mhz")
    if not inst or not mhz:
        return None
    achieved = inst / (eval_ms * 1e-3)
    peak = 4.0 * sms * mhz * 1e6
    return {"bound": "issue", "achieved": achieved, "peak": peak, "unit": "warp instructions/s",
            "frac": achieved / peak, "warp_instructions": inst, "sms": sms, "sm_mhz": mhz}


def reclaim_timing(wf, ctx, dp, res_lru, P, stream, flush):
    """The same batch under reclamation by next use: eval time (next-use pass
    included) and the batch's mean makespan and GPU time against LRU."""
    import torch
    lru = [t.clone() for t in (res_lru.makespan, res_lru.gpu, res_lru.status)]
    wf.wf_ctx_set_reclaim(ctx, wf.RECLAIM_NEXT_USE)
    res = wf.Results(P, dp.place.device)
    e = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    with torch.cuda.stream(stream):
        wf.wf_eval_plans(ctx, dp, res, stream)
        flush_l2(flush)
        e[0].record(stream)
        wf.wf_eval_plans(ctx, dp, res, stream)
        e[1].record(stream)
    torch.cuda.synchronize()
    wf.wf_ctx_set_reclaim(ctx, wf.RECLAIM_LRU)
    ok = (res.status == 0) & (lru[2] == 0)
    mean = lambda t: float(t[ok].double().mean().item())
    return {"eval_ms": e[0].elapsed_time(e[1]), "plans": P,
            "mean_makespan_us": {"lru": mean(lru[0]), "next_use": mean(res.makespan)},
            "mean_gpu_us": {"lru": mean(lru[1]), "next_use": mean(res.gpu)}}


def phi_timing(wf, ctx, dp, P, k, stream, flush):
    """The batch through wf_eval_plans_phi (Eq. 12's window terms beside the
    metrics) and its top-k by that key: eval time (median of 3, L2 flushed
    before each) and the best plan's (makespan, timely prefetches, lifecycle
    overhead)."""
    import torch
    res = wf.Results(P, dp.place.device)
    timely = torch.empty(P, dtype=torch.int64, device=dp.place.device)
    life = torch.empty_like(timely)
    ids = torch.empty(k, dtype=torch.int32, device=dp.place.device)
    keys = torch.empty((k, 3), dtype=torch.int64, device=dp.place.device)
    ts = []
    with torch.cuda.stream(stream):
        wf.wf_eval_plans_phi(ctx, dp, res, timely, life, stream)
        for _ in range(3):
            e = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            flush_l2(flush)
            e[0].record(stream)
            wf.wf_eval_plans_phi(ctx, dp, res, timely, life, stream)
            e[1].record(stream)
            ts.append(e)
        wf.wf_topk_phi(ctx, res, timely, life, P, k, ids, keys, stream)
    torch.cuda.synchronize()
    ms = float(np.median([a.elapsed_time(b) for a, b in ts]))
    best = keys[0].tolist()
    return {"eval_ms": ms, "plans_per_s": P / (ms * 1e-3),
            "best": {"makespan_us": best[0], "timely_prefetches": best[1], "life_us": best[2]}}


# Fixed oracle samples of the other windows (plans), each a few seconds of
# one host thread at most.
OTHER_WORKLOADS = {"tiny": 1024, "mix": 1024, "stochastic": 16, "large": 128}


def workload_entry(name, wf, dev, steps=5, warmup=3, with_cpu=True):
    """One forecast / eval / top-k step of another named window at its full
    size, timed like the headline (CUDA events, L2 flushed before each step),
    with the oracle on a fixed sample of the same batch and the clocks seen.
    Stochastic windows report simulations (plans x samples) per second."""
    import torch

    import wfgen
    w = wfgen.config(name)
    prob, P, k = w.problem, w.P, w.k
    plans = wfgen.make_plans(prob, P, w.plan_seed)
    ctx = wf.Ctx(prob, max_P=P, device=dev.index)
    dp = wf.DevicePlans.from_host(plans, dev)
    res = wf.Results(P, dev)
    rel = torch.empty(prob.N, dtype=torch.int64, device=dev)
    comp = torch.empty_like(rel)
    ids = torch.empty(k, dtype=torch.int32, device=dev)
    keys = torch.empty((k, 3), dtype=torch.int64, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    stream = torch.cuda.Stream(device=dev)
    side = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            flush_l2(flush)
            run_step(wf, ctx, dp, res, rel, comp, ids, keys, P, k, stream, side)
    wf.wf_ctx_status(ctx, stream)
    clocks = ClockSampler(dev.index)
    clocks.start()
    time.sleep(0.2)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(steps)]
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for e in ev:
            flush_l2(flush)
            run_step(wf, ctx, dp, res, rel, comp, ids, keys, P, k, stream, side, e)
    torch.cuda.synchronize()
    clk = clocks.stop()
    wf.wf_ctx_status(ctx, stream)
    step_ms = float(np.median([e[0].elapsed_time(e[3]) for e in ev]))
    eval_ms = float(np.median([e[1].elapsed_time(e[2]) for e in ev]))
    peak = read_peaks().get("hbm_gbs")
    bpp = algorithmic_bytes_per_plan(prob.N)
    entry = {"description": w.description, "P": P, "N": prob.N, "D": prob.D, "k": k,
             "step_ms": step_ms, "eval_ms": eval_ms, "plans_per_s": P / (step_ms * 1e-3),
             "roofline": {"bound": "alu" if prob.S else "hbm",
                          "achieved_gbs": bpp * P / (eval_ms * 1e-3) / 1e9, "peak_gbs": peak,
                          "frac_of_hbm": bpp * P / (eval_ms * 1e-3) / 1e9 / peak if peak else None,
                          "algorithmic_bytes_per_plan": bpp},
             "clocks": clk, "timing": f"median of {steps} steps after {warmup}, L2 flushed before each"}
    traffic, _ = read_traffic(name)
    entry["roofline"]["traffic"] = traffic
    entry["roofline_issue"] = issue_roofline(eval_ms, clk, torch.cuda.get_device_properties(dev).multi_processor_count,
                                             name)
    if prob.S:
        entry["samples"] = prob.S
        entry["sims_per_s"] = P * prob.S / (step_ms * 1e-3)
        ri = entry["roofline_issue"]
        if ri:  # the sims/s this instruction count would give at the full issue rate
            ri["sims_per_s_ceiling"] = P * prob.S / (ri["warp_instructions"] / ri["peak"])
    if with_cpu:
        import oracle
        oracle.build()
        n = min(P, OTHER_WORKLOADS[name])
        t0 = time.perf_counter()
        oracle.eval_plans(prob, plans, 0, n)
        dt = time.perf_counter() - t0
        entry["cpu_baseline"] = {"value": n / dt, "unit": "plans/s", "cores": 1, "kind": "oracle",
                                 "sample": f"the first {n} plans of the {name} batch, one thread, {dt:.2f} s"}
        if prob.S:
            entry["cpu_baseline"]["sims_per_s"] = n * prob.S / dt
    ctx.close()
    del dp, res, plans
    torch.cuda.empty_cache()
    return entry


def batch_timing(wf, prob, dp, P, dev, flush, limits=(1, 2, 4), reps=3):
    """The batch under the replica batch limit B_q (wf_ctx_set_batch, the
    int64 path): eval time (median of reps, L2 flushed before each) and the
    mean makespan and GPU time of the valid plans per limit."""
    import torch
    ctx = wf.Ctx(prob, max_P=P, device=dev.index)
    res = wf.Results(P, dev)
    out = {}
    for B in limits:
        wf.wf_ctx_set_batch(ctx, B)
        ts = []
        for _ in range(reps):
            flush_l2(flush)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            wf.wf_eval_plans(ctx, dp, res)
            b.record()
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        wf.wf_ctx_status(ctx)
        mk, _, gpu, st = res.numpy()
        ok = st == 0
        out[str(B)] = {"eval_ms": float(np.median(ts)), "plans_per_s": P / (float(np.median(ts)) * 1e-3),
                       "mean_makespan_us": float(mk[ok].mean()), "mean_gpu_us": float(gpu[ok].mean())}
    ctx.close()
    return out


def static_timing(wf, prob, plans, dev, flush, reps=5):
    """wf_eval_plans_static (no context, no allocation) on the largest batch
    of this window its static scratch holds: median of reps calls, L2 flushed
    before each."""
    import re

    import torch
    dprob = wf.DeviceProblem(prob, dev)
    fit = plans.P
    try:
        wf.wf_eval_plans_static(dprob, wf.DevicePlans.from_host(plans, dev), wf.Results(plans.P, dev))
        wf.wf_static_status()
    except wf.WfError as e:
        m = re.search(r"at most (\d+) plans", str(e))
        if not m:
            raise
        fit = int(m.group(1))
    sub = plans.slice(0, fit)
    dp = wf.DevicePlans.from_host(sub, dev)
    out = wf.Results(fit, dev)
    ts = []
    for _ in range(reps):
        flush_l2(flush)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        wf.wf_eval_plans_static(dprob, dp, out)
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b))
    wf.wf_static_status()
    ms = float(np.median(ts))
    return {"plans": fit, "ms": ms, "plans_per_s": fit / (ms * 1e-3),
            "timing": f"median of {reps} calls, L2 flushed before each",
            "note": "the largest batch of this window the 32 MiB static scratch holds; a thread per plan"}


def run_gpu(args, rank, world, local):
    import torch

    import wfgen
    from paper_2609_03335_gb300 import build as pkg_build
    from paper_2609_03335_gb300 import wf
    pkg_build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = wfgen.config(WORKLOAD)
    prob, P, k = w.problem, (args.plans or w.P), w.k
    plans = wfgen.make_plans(prob, P, w.plan_seed, plan_base=rank * P)
    t0 = time.perf_counter()
    ctx = wf.Ctx(prob, max_P=P, device=local)
    torch.cuda.synchronize()
    ctx_ms = (time.perf_counter() - t0) * 1e3
    stream = torch.cuda.Stream(device=dev)
    dp = wf.DevicePlans.from_host(plans, dev)
    res = wf.Results(P, dev)
    rel = torch.empty(prob.N, dtype=torch.int64, device=dev)
    comp = torch.empty_like(rel)
    ids = torch.empty(k, dtype=torch.int32, device=dev)
    keys = torch.empty((k, 3), dtype=torch.int64, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    torch.cuda.synchronize()

    side = torch.cuda.Stream(device=dev)

    def step():
        run_step(wf, ctx, dp, res, rel, comp, ids, keys, P, k, stream, side)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            flush_l2(flush)
            step()
    wf.wf_ctx_status(ctx, stream)

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for s in range(args.steps):
            flush_l2(flush)
            run_step(wf, ctx, dp, res, rel, comp, ids, keys, P, k, stream, side, ev[s])
    torch.cuda.synchronize()
    barrier(world)
    wf.wf_ctx_status(ctx, stream)
    step_ms = [e[0].elapsed_time(e[3]) for e in ev]
    eval_ms = [e[1].elapsed_time(e[2]) for e in ev]
    forecast_ms = float(np.mean([e[4].elapsed_time(e[5]) for e in ev]))
    topk_ms = float(np.mean([e[2].elapsed_time(e[3]) for e in ev]))
    ms_per_step = max_over_ranks(float(np.mean(step_ms)), world)
    eval_ms_mean = float(np.mean(eval_ms))

    # End to end through the host-memory call: every step hands wf_eval_topk_host the batch's
    # page-locked host rows; the library copies them into one of its two staging slots on its own
    # copy stream (overlapping the previous step's evaluation, as a serving loop would run),
    # forecasts, evaluates, selects the top-k and copies the top-k and the forecast back into
    # page-locked host memory.  Every step's copies lie inside the timed region.
    hplans = wf.DevicePlans.host(plans)
    hplans.plan_base = rank * P
    pad = lambda b: (b + 15) // 16 * 16
    h2d = P * (pad(prob.N) + pad(2 * prob.N) + 2 * pad(4 * ((prob.N + 31) // 32)))
    ids_h = torch.empty(k, dtype=torch.int32).pin_memory()
    keys_h = torch.empty((k, 3), dtype=torch.int64).pin_memory()
    rel_h = torch.empty(prob.N, dtype=torch.int64).pin_memory()
    comp_h = torch.empty(prob.N, dtype=torch.int64).pin_memory()
    d2h = ids_h.numel() * 4 + keys_h.numel() * 8 + 2 * prob.N * 8
    wf.wf_ctx_reserve_host(ctx)

    def e2e_step(i):
        wf.wf_eval_topk_host(ctx, hplans, k, ids_h, keys_h, None, rel_h, comp_h, stream)

    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            e2e_step(i)
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)  # (the stream is idle: the first step's copy starts after this)
        for i in range(args.steps):
            e2e_step(i)
        e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    # before the search rewrites rows 0..31; the policy needs deterministic latencies
    nextuse = reclaim_timing(wf, ctx, dp, res, P, stream, flush) if prob.S == 0 else None
    phi = phi_timing(wf, ctx, dp, P, k, stream, flush) if prob.S == 0 else None
    search = local_search_timing(wf, ctx, dp, prob, P, stream, flush, peak_gbs=read_peaks().get("hbm_gbs"))
    built = construct_timing(wf, ctx, prob, P, k, stream, flush, random_best=int(keys[0, 0].item()))
    clk = clocks.stop()
    static = static_timing(wf, prob, plans, dev, flush) if prob.S == 0 and world == 1 else None
    batched = batch_timing(wf, prob, dp, P, dev, flush) if prob.S == 0 and world == 1 else None
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    # the host reads the top-k it copied back
    assert int(ids_h.numpy().min()) >= 0

    bpp = algorithmic_bytes_per_plan(prob.N)
    achieved = bpp * P / (eval_ms_mean * 1e-3) / 1e9
    peaks = read_peaks()
    peak = peaks.get("hbm_gbs")
    traffic, _ = read_traffic(WORKLOAD)
    # forecast, status, 32-bit sweep, 64-bit sweep over its hand-offs, int64
    # pass over what is left, top-k passes (the count reset is a memset and
    # the count read-back a copy, not kernels)
    # (stochastic latencies: forecast, status, sample sweep, int64 pass over
    # its hand-offs, top-k passes)
    launches = args.steps * ((5 if prob.S == 0 else 4) + topk_launches(P, k))

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        sample = P if WORKLOAD == "burst" else min(P, 1024)
        t0 = time.perf_counter()
        oracle.eval_plans(prob, plans, 0, sample)
        dt = time.perf_counter() - t0
        cpu = {"value": sample / dt, "unit": "plans/s", "cores": 1, "kind": "oracle",
               "sample": f"{'all' if sample == P else 'the first'} {sample} plans of the {WORKLOAD} batch, "
                         f"one thread, {dt:.2f} s", **host_cpu()}

    if rank == 0:
        line = {
            "metric": metric_of(prob), "value": P * world / (ms_per_step * 1e-3), "unit": "plans/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
            "data": "synthetic",
            "config": {"workload": f"{WORKLOAD}: {w.description} plans per GPU (here {P}), k={k}",
                       "P_per_gpu": P, "N": prob.N, "k": k,
                       "l2": "flushed between timed steps (256 MiB write, then read back)",
                       "ctx_create_ms": ctx_ms,
                       "stage_ms": {"forecast": forecast_ms, "eval": eval_ms_mean, "topk": topk_ms}},
            "e2e": {"value": P * world / (e2e_ms * 1e-3), "unit": "plans/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak if peak else None,
                         "traffic": traffic,
                         "kernel": ("wf_eval_plans = status_kernel + pc_kernel (u32 times) + pc_kernel (u64 "
                                    "times, hand-offs) + eval_list_kernel") if prob.S == 0 else
                                   "wf_eval_plans = status_kernel + stoch_kernel + eval_stoch_kernel (hand-offs)",
                         "algorithmic_bytes_per_plan": bpp, "kernel_ms": eval_ms_mean,
                         "peak_source": "MEASURED_PEAKS.json hbm_gbs (measured copy)" if peak else None},
            "roofline_issue": issue_roofline(eval_ms_mean, clk, torch.cuda.get_device_properties(dev).multi_processor_count),
            "cpu_baseline": cpu,
            "clocks": clk,
            "gpu_launches": launches,
            "local_search": search,
            "construct": built,
            "reclaim_next_use": nextuse,
            "eq12_window_terms": phi,
            "static_entry": static,
            "replica_batch": batched,
        }
        if world == 1 and not args.no_workloads and WORKLOAD == "burst":
            # the other named windows, each at its full size (context, plans
            # and L2 flush of their own)
            del dp, res
            torch.cuda.empty_cache()
            line["workloads"] = {n: workload_entry(n, wf, dev, with_cpu=not args.no_cpu_baseline)
                                 for n in OTHER_WORKLOADS}
        print(json.dumps(line), flush=True)
    ctx.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("gpu", "reference"), default="gpu")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-workloads", action="store_true", help="skip the other named windows")
    ap.add_argument("--workload", default="burst", choices=("tiny", "mix", "burst", "stochastic", "large"),
                    help="the synthetic window (burst is the headline configuration)")
    ap.add_argument("--plans", type=int, default=0, help="plans per GPU (default: the workload's)")
    args = ap.parse_args()
    global WORKLOAD
    WORKLOAD = args.workload
    rank, world, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, rank, world)
    else:
        run_gpu(args, rank, world, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
