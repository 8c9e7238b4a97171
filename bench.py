"""Benchmark: scheduled denoiser steps/s at a layer-step budget on one GB300.

Default workload: the LLaDA-8B-shaped masked-diffusion transformer (32 blocks,
d 4096, 32 heads x 128, SwiGLU 12288, RMSNorm, RoPE, 126464-token head), batch 4 x
1024 tokens, horizon T = 64, 50% layer-step budget from the SCR/Frobenius
schedule.  A bench "step" is one denoiser evaluation (one sgd_step: stem, every
active unit, frozen runs, head) at trajectory position s.  The K timed steps are
K // T whole trajectories plus, when K is not a multiple of T, K % T positions
spread evenly over 1..T (the midpoints of K % T equal slices); every trajectory
runs in order from s = 1 (the untimed steps in between fill the caches), and
each run of consecutive timed steps sits between its own pair of CUDA events.

Prints ONE JSON line (rank 0).  --impl reference times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "scheduled denoiser steps/s at 50% layer-step budget; % of BF16/HBM roofline"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None, help="timed denoiser steps (default T)")
    ap.add_argument("--warmup", type=int, default=None, help="untimed steps (default T)")
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--config", default="llada")
    ap.add_argument("--budget", type=float, default=0.5)
    ap.add_argument("--T", type=int, default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="also time one trajectory at 100/50/33%% budgets (adds key 'budget_sweep')")
    ap.add_argument("--ablation", action="store_true",
                    help="also time the execution modes of Table tab:kernel (adds key 'ablation')")
    ap.add_argument("--rankings", action="store_true",
                    help="also time one trajectory per static ranking of Table tab:cross-ablation "
                         "and for branch granularity, all at the same budget (adds key 'rankings')")
    ap.add_argument("--flags", type=int, default=0,
                    help="sgd_model_desc flags for ablations (e.g. 16: programmatic dependent "
                         "launch, 32: pre-norms folded into the GEMMs)")
    ap.add_argument("--policies", action="store_true",
                    help="also time the static schedule against the activation-drift policy of "
                         "App. B.1 at the same budget (adds key 'policies')")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d["bf16_tflops_sustained"],
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms while running."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        loaded = [x for x in sm if x > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(n_gpus):
    """Rank, world size and local rank from the launcher's environment; for N > 1 one process
    group over NCCL (gloo when no GPU is visible, as in the CPU tests of this path)."""
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """The largest of every rank's x (the slowest rank's time sets the job's time)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# workload
# ---------------------------------------------------------------------------

def timed_plan(K, T):
    """Trajectories of the timed region and, for each, its timed positions (1-based, in
    order): K // T whole trajectories, then the midpoints of K % T equal slices of 1..T,
    so that the timed steps sample the whole horizon and its active-set profile."""
    full, rem = divmod(K, T)
    plan = [list(range(1, T + 1)) for _ in range(full)]
    if rem:
        plan.append([int((i + 0.5) * T / rem) + 1 for i in range(rem)])
    return plan


def golden_module():
    """tests/golden/full_size_schedules.py: the oracle's stored full-size schedules."""
    import importlib.util
    path = os.path.join(ROOT, "tests", "golden", "full_size_schedules.py")
    spec = importlib.util.spec_from_file_location("sgd_full_size_schedules", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def setup_workload(args, device):
    import torch
    from paper_2609_29505_gb300 import schedule, synth
    cfg = synth.get_config(args.config)
    T = args.T or cfg.T
    t0 = time.time()
    weights = synth.make_weights(cfg, device)
    inp = synth.make_inputs(cfg, device)
    if str(device).startswith("cuda"):
        torch.cuda.synchronize()
    t_w = time.time() - t0
    t0 = time.time()
    sched = schedule.build_schedule(cfg, weights, T, budget=args.budget)
    t_s = time.time() - t0
    return cfg, T, weights, inp, sched, dict(weights_s=round(t_w, 1), schedule_s=round(t_s, 1))


def step_inputs(cfg, inp, T, device):
    """Per-step device inputs for positions s = 1..T (token models: reveal schedule;
    continuous models: the seeded initial state, held fixed)."""
    import torch
    from paper_2609_29505_gb300 import synth
    if cfg.stem == "embed":
        return [synth.token_ids_at(cfg, inp, s, T).to(device).contiguous() for s in range(1, T + 1)]
    z = inp.z0.to(device).contiguous()
    return [z for _ in range(T)]


def out_buffer(cfg, device, pinned=False):
    import torch
    if cfg.head == "logits":
        shape, dt = (cfg.batch, cfg.n_tokens, cfg.d_out), torch.float16
    elif cfg.head == "identity":
        shape, dt = (cfg.batch, cfg.n_tokens, cfg.d), torch.float32
    else:
        shape, dt = (cfg.batch, cfg.n_out_tokens, cfg.out_channels), torch.float32
    if device == "cpu":
        t = torch.empty(shape, dtype=dt)
        return t.pin_memory() if pinned else t
    return torch.empty(shape, dtype=dt, device=device)


def run_native(args):
    import torch
    from paper_2609_29505_gb300 import binding, build

    build.build()
    rank, world, local = dist_setup(args.gpus)
    dev = torch.device("cuda", local if world > 1 else 0)
    peaks = load_peaks()
    cfg, T, weights, inp, sched, setup_t = setup_workload(args, dev)
    K = args.steps if args.steps is not None else T
    W = args.warmup if args.warmup is not None else T
    W = max(W, 3)
    model = binding.Denoiser(cfg, weights, flags=args.flags)
    t0 = time.time()
    model.set_schedule(T, sched["lifetimes"], sched["groups"])
    setup_t["capture_s"] = round(time.time() - t0, 2)
    info = model.info()
    xs = step_inputs(cfg, inp, T, dev)
    cls = None if inp.class_ids is None else inp.class_ids.to(dev)
    ctx = None if inp.ctx is None else inp.ctx.to(dev)
    out = out_buffer(cfg, dev)
    stream = torch.cuda.current_stream()
    from paper_2609_29505_gb300.synth import timestep

    def run_steps(n, start_fresh=True):
        if start_fresh:
            model.reset()
        for i in range(n):
            s = i % T + 1
            model.step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls, ctx=ctx, stream=stream)

    run_steps(W)
    torch.cuda.synchronize()
    model.check_device(stream)
    # timed region: exactly K steps (timed_plan), CUDA events around each run of
    # consecutive timed steps; untimed steps between them only fill the caches
    plan = timed_plan(K, T)
    timed_pos = [s for traj in plan for s in traj]
    barrier(world)
    torch.cuda.synchronize()
    pairs = []
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index if dev.index is not None else 0) as clk:
        w0.record(stream)
        for traj in plan:
            model.reset()
            tset = set(traj)
            for s in range(1, max(traj) + 1):
                if s in tset and s - 1 not in tset:
                    e0 = torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                model.step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls, ctx=ctx, stream=stream)
                if s in tset and s + 1 not in tset:
                    e1 = torch.cuda.Event(enable_timing=True)
                    e1.record(stream)
                    pairs.append((e0, e1))
        w1.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms = sum(a.elapsed_time(b) for a, b in pairs)
    ms = max_over_ranks(ms, world)
    region_ms = w0.elapsed_time(w1)
    model.check_device(stream)
    value = K * world / (ms / 1000.0)
    n_groups = len(set(sched["groups"]))
    group_S = {}
    for g, S_u in zip(sched["groups"], sched["lifetimes"]):
        group_S[int(g)] = int(S_u)
    timed_ratio = sum(sum(1 for S_g in group_S.values() if S_g >= s) for s in timed_pos) / (K * n_groups)

    # per-op timing of one trajectory (same kernels, launched op by op with events)
    recs_by_step = []
    model.reset()
    for s in range(1, T + 1):
        recs_by_step.append(model.profile_step(xs[s - 1], out, timestep(cfg, s, T), s,
                                               class_ids=cls, ctx=ctx, stream=stream))
    launches_per_pos = [len(r) + 1 for r in recs_by_step]  # + the per-step I/O-slot kernel
    gpu_launches = sum(launches_per_pos[s - 1] for s in timed_pos)
    if cfg.block == "xattn":
        gpu_launches += cfg.n_blocks * timed_pos.count(1)  # context K/V at each timed s = 1
    # per-kernel sums over exactly the timed positions (with their multiplicity)
    by_kernel = {}
    tot_flops = tot_bytes = tot_ms = 0.0
    t_roof_timed = 0.0
    for s in timed_pos:
        recs = recs_by_step[s - 1]
        fl_s = sum(r["flops"] for r in recs)
        by_s = sum(r["bytes"] for r in recs)
        t_roof_timed += max(fl_s / (peaks["bf16_sus"] * 1e12), by_s / (peaks["hbm"] * 1e9))
        for r in recs:
            k = by_kernel.setdefault(r["kernel"], dict(ms=0.0, flops=0.0, bytes=0.0, launches=0))
            k["ms"] += r["ms"]
            k["flops"] += r["flops"]
            k["bytes"] += r["bytes"]
            k["launches"] += 1
            tot_flops += r["flops"]
            tot_bytes += r["bytes"]
            tot_ms += r["ms"]
    gemm = by_kernel.get("gemm_tc", by_kernel.get("gemm_simt"))
    achieved = gemm["flops"] / (gemm["ms"] / 1e3) / 1e12
    roofline = {"bound": "tensor", "kernel": "gemm_tcgen05", "achieved": round(achieved, 1),
                "peak": peaks["bf16_sus"], "unit": "TFLOP/s",
                "frac": round(achieved / peaks["bf16_sus"], 4),
                "peak_source": f"{peaks['source']} bf16 sustained x 1 (fp16 and bf16 share the "
                               "kind::f16 dense rate)", "traffic": gemm_traffic(cfg, T, args.budget),
                "traffic_unit": "DRAM bytes per launch (ncu, one cold launch of each GEMM of the step, "
                                "averaged with the step's launch mix; profiles/gemm_tcgen05_llada_dram.md)",
                "algorithmic_bytes_per_launch": round(gemm["bytes"] / gemm["launches"]),
                "launches_in_timed_steps": gemm["launches"],
                "measured_over": "the timed positions, one eager op-by-op launch per op with "
                                 "CUDA events (same kernels and launch configurations as the graphs)",
                "share_of_step": round(gemm["ms"] / tot_ms, 3)}
    fz = by_kernel.get("frozen_run")
    # step roofline over exactly the timed steps: sum over them of max(FLOPs / bf16 peak,
    # bytes / HBM peak), against their measured time
    traj_fl = sum(r["flops"] for recs in recs_by_step for r in recs)
    traj_by = sum(r["bytes"] for recs in recs_by_step for r in recs)
    t_roof_traj = sum(max(sum(r["flops"] for r in recs) / (peaks["bf16_sus"] * 1e12),
                          sum(r["bytes"] for r in recs) / (peaks["hbm"] * 1e9)) for recs in recs_by_step)
    step_roof = {"t_roofline_ms": round(t_roof_timed * 1e3 / K, 3), "t_measured_ms": round(ms / K, 3),
                 "frac": round(t_roof_timed * 1e3 / ms, 4),
                 "flops_per_step": tot_flops / K, "bytes_per_step": tot_bytes / K,
                 "roofline_steps_per_s": round(K / t_roof_timed, 2),
                 "over": "the K timed steps",
                 "trajectory": {"flops_per_step": traj_fl / T, "bytes_per_step": traj_by / T,
                                "roofline_steps_per_s": round(T / t_roof_traj, 2)}}
    kernels = {k: {"launches": v["launches"], "ms_in_timed_steps": round(v["ms"], 3),
                   "share": round(v["ms"] / tot_ms, 4),
                   "tflops": round(v["flops"] / max(v["ms"], 1e-9) / 1e9, 1),
                   "gbs": round(v["bytes"] / max(v["ms"], 1e-9) / 1e6, 1)} for k, v in by_kernel.items()}
    if fz:
        kernels["frozen_run"]["frac_of_hbm"] = round(fz["bytes"] / (fz["ms"] / 1e3) / 1e9 / peaks["hbm"], 4)

    # end to end through the C ABI with host buffers (pinned): every step copies its
    # inputs in and its whole output back (pinned output buffers: the step's output kernel
    # writes them directly over the host link)
    e2e = None
    if not args.no_e2e:
        import torch as _t
        xs_h = [x.cpu().pin_memory() for x in xs[:T]]
        outs_h = [out_buffer(cfg, "cpu", pinned=True) for _ in range(2)]
        cls_h = None if inp.class_ids is None else inp.class_ids.cpu().pin_memory()
        ctx_h = None if inp.ctx is None else inp.ctx.cpu().pin_memory()
        n_e2e = len(plan) * T  # whole trajectories: every step of each, in order
        barrier(world)
        _t.cuda.synchronize()
        with ClockSampler(dev.index if dev.index is not None else 0) as clk_e2e:
            t0 = time.perf_counter()
            for i in range(n_e2e):
                s = i % T + 1
                if s == 1:
                    model.reset()
                model.step_host_async(xs_h[s - 1], outs_h[i % 2], timestep(cfg, s, T), s,
                                      class_ids_host=cls_h, ctx_host=ctx_h, stream=stream)
            model.host_wait()
            _t.cuda.synchronize()
            e2e_s = max_over_ranks(time.perf_counter() - t0, world)
        h2d = xs_h[0].numel() * xs_h[0].element_size() + (0 if cls_h is None else cls_h.numel() * 4)
        e2e = {"value": round(n_e2e * world / e2e_s, 3), "unit": "steps/s", "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(outs_h[0].numel() * outs_h[0].element_size()),
               "steps": n_e2e, "over": f"{len(plan)} whole trajectory(ies) of T={T} steps",
               "clocks": clk_e2e.summary(),
               "api": "sgd_step_host_async + sgd_host_wait (pinned host output written by the step's output kernel)"}

    sweep = None
    if args.sweep:
        sweep = run_sweep(binding, model, cfg, T, weights, sched, xs, out, cls, ctx, stream, peaks)

    ablation = None
    if args.ablation:
        ablation = run_ablation(binding, model, cfg, T, weights, sched, xs, out, cls, ctx, stream)

    rankings = None
    if args.rankings:
        rankings = run_rankings(binding, model, cfg, T, weights, args.budget, sched, xs, out, cls,
                                ctx, stream)

    policies = None
    if args.policies:
        policies = run_policies(binding, model, cfg, T, xs, out, cls, ctx, stream)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, T, weights, inp, args.budget, n_steps=8)

    model.close()
    res = {
        "metric": METRIC if args.budget == 0.5 else METRIC.replace("50%", f"{args.budget:.0%}"),
        "value": round(value, 3), "unit": "steps/s", "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": round(ms / K, 3), "higher_is_better": True, "scaling": "weak",
        "timed_positions": timed_pos if len(timed_pos) <= 256 else None,
        "timed_layer_step_ratio": round(timed_ratio, 4),
        "timed_region_ms": round(region_ms, 2),
        "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "precision": "fp16 operands (bf16 weights converted exactly, power-of-two scaled), "
                     "fp32 accumulation and fp32 residual stream",
        "config": {"workload": workload_name(cfg, T, args.budget), "batch": cfg.batch,
                   "seq_len": cfg.n_tokens, "T": T, "budget": args.budget,
                   "achieved_layer_step_ratio": round(sched["ratio"], 4),
                   "tokens_per_s": round(value * cfg.batch * cfg.n_tokens, 1),
                   "parallelism": f"replicas{world}" if world > 1 else "single",
                   "l2": "inputs larger than L2 (bf16 weights ~16 GB per step)",
                   "n_patterns": info["n_patterns"], "n_graphs": info["n_graphs"], "flags": args.flags,
                   "cache_gb": round(info["cache_bytes"] / 2 ** 30, 2), "setup": setup_t},
        "roofline": roofline, "step_roofline": step_roof, "kernels": kernels,
        "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": int(gpu_launches),
        "ablation": ablation, "budget_sweep": sweep, "policies": policies, "rankings": rankings,
        "clocks": clk.summary(),
    }
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_sweep(binding, model, cfg, T, weights, sched, xs, out, cls, ctx, stream, peaks):
    """One trajectory per budget (same weights and inputs): steps/s, tokens/s, and the
    step roofline from the per-op records of one profiled trajectory."""
    import torch
    from paper_2609_29505_gb300 import schedule
    from paper_2609_29505_gb300.synth import timestep
    rows = []
    bq = sched["branch_scores"]
    for budget in (1.0, 0.5, 0.33):
        sc = schedule.build_schedule(cfg, weights, T, budget=budget, branch_q=bq)
        model.set_schedule(T, sc["lifetimes"], sc["groups"])
        for rep in range(2):
            model.reset()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for s in range(1, T + 1):
                model.step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls, ctx=ctx, stream=stream)
            e1.record(stream)
            torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        model.reset()
        fl = by = 0.0
        for s in range(1, T + 1):
            for r in model.profile_step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls,
                                        ctx=ctx, stream=stream):
                fl += r["flops"]
                by += r["bytes"]
        t_roof = max(fl / (peaks["bf16_sus"] * 1e12), by / (peaks["hbm"] * 1e9))
        sps = T / (ms / 1e3)
        rows.append({"budget": budget, "achieved_ratio": round(sc["ratio"], 4),
                     "steps_per_s": round(sps, 2), "tokens_per_s": round(sps * cfg.batch * cfg.n_tokens, 1),
                     "ms_per_step": round(ms / T, 3), "roofline_steps_per_s": round(T / t_roof, 2),
                     "roofline_frac": round(t_roof * 1e3 / ms, 4)})
    model.set_schedule(T, sched["lifetimes"], sched["groups"])
    return rows


def run_ablation(binding, model, cfg, T, weights, sched, xs, out, cls, ctx, stream):
    """Execution modes of Table tab:kernel on this workload: eager full inference (100%
    schedule, one launch per op), host-side skipping (budget schedule, eager), padded
    static graphs (every frozen branch still evaluated) and jagged graphs.  One whole
    trajectory each, CUDA events on the stream."""
    import torch
    from paper_2609_29505_gb300.synth import timestep
    full = [T] * cfg.n_units
    rows = []
    modes = [("eager_full", full, binding.EXEC_EAGER),
             ("host_skipping", sched["lifetimes"], binding.EXEC_EAGER),
             ("padded_graph", sched["lifetimes"], binding.EXEC_PADDED_GRAPH),
             ("jagged_graph", sched["lifetimes"], binding.EXEC_JAGGED_GRAPH)]
    for name, S, mode in modes:
        model.set_schedule(T, S, sched["groups"])
        model.set_exec_mode(mode)
        for rep in range(2):  # first pass warms the mode up
            model.reset()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for s in range(1, T + 1):
                model.step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls, ctx=ctx, stream=stream)
            e1.record(stream)
            torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        executed = cfg.n_blocks * T if mode == binding.EXEC_PADDED_GRAPH else int(sum(S)) // len(cfg.branches)
        rows.append({"mode": name, "trajectory_ms": round(ms, 2), "layer_steps_executed": executed})
    model.set_exec_mode(binding.EXEC_JAGGED_GRAPH)
    model.set_schedule(T, sched["lifetimes"], sched["groups"])
    base = rows[0]["trajectory_ms"]
    for r in rows:
        r["speedup_vs_eager_full"] = round(base / r["trajectory_ms"], 3)
    return rows


def run_rankings(binding, model, cfg, T, weights, budget, sched, xs, out, cls, ctx, stream):
    """Latency of the alternative static rankings (Table tab:cross-ablation) and of branch
    granularity at the same layer-step budget: the same kernels run; what changes is which
    units are active at each step, hence the active patterns and graphs.  One trajectory
    each after a warm-up trajectory, CUDA events on the stream."""
    import torch
    from paper_2609_29505_gb300 import schedule
    from paper_2609_29505_gb300.synth import timestep
    rows = []
    variants = [(r, "block") for r in ("scr", "frobenius", "spectral", "stable_rank",
                                       "frob_stable_rank", "raw_scr", "depth", "random")]
    variants.append(("scr", "branch"))
    for ranking, gran in variants:
        sc = schedule.build_schedule(cfg, weights, T, budget=budget, ranking=ranking, granularity=gran)
        model.set_schedule(T, sc["lifetimes"], sc["groups"])
        for rep in range(2):
            model.reset()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for s in range(1, T + 1):
                model.step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls, ctx=ctx, stream=stream)
            e1.record(stream)
            torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        info = model.info()
        rows.append({"ranking": ranking, "granularity": gran, "achieved_ratio": round(sc["ratio"], 4),
                     "n_patterns": info["n_patterns"], "trajectory_ms": round(ms, 2),
                     "steps_per_s": round(T / (ms / 1e3), 3)})
    model.set_schedule(T, sched["lifetimes"], sched["groups"])
    return rows


def run_policies(binding, model, cfg, T, xs, out, cls, ctx, stream):
    """Latency side of Table tab:input-aware: whole trajectories under the static schedule
    and under the causal activation-drift policy (same per-step active counts; drift
    reductions, host routing after every step, graph lookup and eager fallback included).
    Two trajectories each after one warm-up trajectory, CUDA events on the stream."""
    import torch
    from paper_2609_29505_gb300.synth import timestep
    rows = {}
    for name, pol in (("static", binding.POLICY_STATIC), ("drift", binding.POLICY_DRIFT)):
        model.set_policy(pol)
        i0 = model.info()
        times = []
        for rep in range(3):  # the first pass warms the policy up
            model.reset()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for s in range(1, T + 1):
                model.step(xs[s - 1], out, timestep(cfg, s, T), s, class_ids=cls, ctx=ctx, stream=stream)
            e1.record(stream)
            torch.cuda.synchronize()
            if rep:
                times.append(e0.elapsed_time(e1))
        i1 = model.info()
        ms = sum(times) / len(times)
        rows[name] = {"trajectory_ms": round(ms, 2), "steps_per_s": round(T / (ms / 1e3), 3)}
        if pol == binding.POLICY_DRIFT:
            rows[name]["graph_steps"] = int(i1["graph_steps"] - i0["graph_steps"])
            rows[name]["eager_steps"] = int(i1["eager_steps"] - i0["eager_steps"])
    model.set_policy(binding.POLICY_STATIC)
    rows["drift_slowdown"] = round(rows["drift"]["trajectory_ms"] / rows["static"]["trajectory_ms"], 3)
    return rows


GEMM_SOURCES = ("gemm_kernel.cuh", "gemm.cu", "common.cuh")


def gemm_source_hash():
    import hashlib
    h = hashlib.sha256()
    for f in GEMM_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_29505_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def gemm_traffic(cfg, T, budget):
    """DRAM bytes per GEMM launch (read + write, averaged over the step's GEMM launches) from
    the committed ncu summary of this workload's GEMMs, or None when the workload differs or
    the GEMM sources changed since the counters were taken."""
    import re
    path = os.path.join(ROOT, "profiles", "gemm_tcgen05_llada_dram.md")
    if cfg.name != "llada" or T != 64 or abs(budget - 0.5) > 1e-9 or not os.path.exists(path):
        return None
    m = re.search(r"traffic_bytes_per_launch: (\d+) sources: ([0-9a-f]{16})", open(path).read())
    if not m:
        return None
    return int(m.group(1)) if gemm_source_hash() == m.group(2) else None


def workload_name(cfg, T, budget):
    names = {"llada": "LLaDA-8B-shaped", "dit": "DiT-XL/2-shaped", "uvit": "U-ViT-L-shaped",
             "sdxl": "SDXL-transformer-shaped", "tiny": "tiny pre-norm",
             "llada_4k": "LLaDA-8B-shaped 4K-context"}
    return (f"{names.get(cfg.name, cfg.name)} B={cfg.batch} N={cfg.n_tokens} d={cfg.d} "
            f"L={cfg.n_blocks} T={T} budget={budget:.0%}")


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------

TOKEN_SAMPLE = 128


def token_model_flops(cfg, n_active_blocks, batch, n_tokens):
    """Dense FLOPs of one step of a token (pre-norm, gated-MLP) model with n_active_blocks
    active blocks: per active block QKV, attention output, up and down projections
    (2 n params) and non-causal attention (4 n^2 d); the vocabulary head at every step."""
    d, f = cfg.d, cfg.d_ff
    per_block = 2 * n_tokens * (4 * d * d + 3 * d * f) + 4 * n_tokens * n_tokens * d
    return batch * (n_active_blocks * per_block + 2 * n_tokens * d * cfg.d_out)


def oracle_sample(cfg, T, weights, inp):
    """Bounded sample of the workload for the CPU oracle: batch row 0 and, for token
    models, its first TOKEN_SAMPLE positions (full depth, width and head).  Returns the
    oracle model config, fp32 weights, a state function, a function giving the workload's
    FLOPs over the sample's FLOPs for a list of (position, active blocks), the class ids,
    the context and a description."""
    from paper_2609_29505_gb300 import synth
    W = {k: v.detach().float().cpu().numpy() for k, v in weights.items()}
    if cfg.stem == "embed":
        n = min(TOKEN_SAMPLE, cfg.n_tokens)
        ocfg = cfg.with_(batch=1, n_tokens=n)
        state = lambda s: synth.token_ids_at(cfg, inp, s, T)[:1, :n].cpu().numpy()

        def scale(active):
            full = sum(token_model_flops(cfg, a, cfg.batch, cfg.n_tokens) for a in active)
            samp = sum(token_model_flops(cfg, a, 1, n) for a in active)
            return full / samp
        desc = (f"batch row 0 of {cfg.batch}, first {n} of {cfg.n_tokens} tokens, all layers and "
                f"the full head; scaled to the workload by its dense FLOPs (attention quadratic in "
                f"tokens)")
    else:
        ocfg = cfg.with_(batch=1)
        z0 = inp.z0[:1].cpu().numpy()
        state = lambda s: z0
        scale = lambda active: float(cfg.batch)  # samples are independent: exact
        desc = f"batch row 0 of {cfg.batch}, all tokens and layers; scaled by the batch"
    cls = None if inp.class_ids is None else inp.class_ids[:1].cpu().numpy()
    ctx = None if inp.ctx is None else inp.ctx[:1].float().cpu().numpy()
    return ocfg, W, state, scale, cls, ctx, desc


def cpu_threads():
    try:
        import threadpoolctl
        info = threadpoolctl.threadpool_info()
        return max((i.get("num_threads", 1) for i in info), default=os.cpu_count())
    except Exception:
        return os.cpu_count()


def oracle_schedule(cfg, weights, T, budget):
    """Per-unit lifetimes from oracle.spectral (stored for the full-size models, checked
    against the weights' checksum, else computed here) and the active blocks per step."""
    from paper_2609_29505_gb300 import synth
    S, source = golden_module().oracle_lifetimes(cfg, weights, T, budget)
    groups = synth.block_groups(cfg)
    G = max(groups) + 1
    Sg = [0] * G
    for g, x in zip(groups, S):
        Sg[g] = int(x)
    active = lambda s: sum(1 for x in Sg if x >= s)
    return [int(x) for x in S], active, source


def time_oracle(cfg, T, weights, inp, budget, positions, warm_positions=(), octx=None):
    """Wall time of the oracle's scheduled forward on the sample at the given positions."""
    from oracle import trajectory as otj
    ocfg, W, state, scale, cls, ctx, desc = octx or oracle_sample(cfg, T, weights, inp)
    S, active, source = oracle_schedule(cfg, weights, T, budget)
    if warm_positions:
        otj.time_steps(ocfg, W, S, T, list(warm_positions), state, cls, ctx)
    t0 = time.perf_counter()
    otj.time_steps(ocfg, W, S, T, list(positions), state, cls, ctx)
    el = time.perf_counter() - t0
    f = scale([active(s) for s in positions])
    return el, f, desc, source


def cpu_baseline(cfg, T, weights, inp, budget, n_steps=8):
    """Oracle steps/s on the host cores for a bounded sample (about 10-30 s of work), at
    n_steps positions spread over the horizon."""
    positions = timed_plan(min(n_steps, T), T)[0]
    el, f, desc, source = time_oracle(cfg, T, weights, inp, budget, positions)
    per_step = el / len(positions)
    return {"value": round(1.0 / (per_step * f), 6), "unit": "steps/s", "cores": cpu_threads(),
            "kind": "oracle", "sample_s_per_step": round(per_step, 3), "scale": round(f, 4),
            "lifetimes": f"oracle.spectral ({source})",
            "sample": f"{desc}; positions {positions} of T={T}; value = 1 / (sample s/step x scale)"}


def run_reference(args):
    """--impl reference: the CPU oracle timed on the host cores (rank 0 only), at the
    positions the native arm times, with the oracle's own lifetimes.  The synthetic weights
    come from the same seeded generator on the same device as the native arm's (the same
    bytes); nothing of the method runs on the GPU."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch
    from paper_2609_29505_gb300 import synth
    cfg = synth.get_config(args.config)
    T = args.T or cfg.T
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    weights = synth.make_weights(cfg, dev)
    inp = synth.make_inputs(cfg, dev)
    K = args.steps if args.steps is not None else T
    Wm = args.warmup if args.warmup is not None else 1
    positions = [s for traj in timed_plan(K, T) for s in traj]
    warm = [i % T + 1 for i in range(Wm)]
    t0 = time.perf_counter()
    octx = oracle_sample(cfg, T, weights, inp)
    el, f, desc, source = time_oracle(cfg, T, weights, inp, args.budget, positions, warm, octx)
    setup_s = time.perf_counter() - t0 - el
    per_step = el / K
    value = 1.0 / (per_step * f)
    res = {"impl": "reference", "metric": METRIC if args.budget == 0.5 else
           METRIC.replace("50%", f"{args.budget:.0%}"), "value": round(value, 6), "unit": "steps/s",
           "n_gpus": 1, "steps": K, "warmup": Wm,
           "ms_per_step": round(per_step * 1e3, 3),
           "ms_per_step_is": "measured wall time of one sample step (value = 1 / (that x scale))",
           "scale": round(f, 4), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "f32", "data": "synthetic", "timed_positions": positions if K <= 256 else None,
           "config": {"workload": workload_name(cfg, T, args.budget), "batch": cfg.batch,
                      "seq_len": cfg.n_tokens, "T": T, "budget": args.budget},
           "setup_s": round(setup_s, 1),
           "cpu_baseline": {"value": round(value, 6), "unit": "steps/s", "cores": cpu_threads(),
                            "kind": "oracle", "sample_s_per_step": round(per_step, 3),
                            "scale": round(f, 4), "lifetimes": f"oracle.spectral ({source})",
                            "sample": desc},
           "e2e": {"value": round(value, 6), "unit": "steps/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(res), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
