"""Single-kernel cases of libsgd at the LLaDA-8B-shaped sizes, timed with CUDA events.

Each case launches one hot-path kernel through the C ABI (include/sgd_kernels.h)
with the same launch configuration sgd_step uses, on inputs larger than L2, and
prints one JSON line: average launch time and achieved TFLOP/s or GB/s.  It is the
command that the committed ncu summaries under profiles/ were captured from.

    python -m paper_2609_29505_gb300.kernel_bench gemm --M 4096 --N 12288 --K 4096 --epi rope
    python -m paper_2609_29505_gb300.kernel_bench attention --batch 4 --heads 32 --tokens 1024 --dh 128
    python -m paper_2609_29505_gb300.kernel_bench attention --batch 8 --heads 16 --tokens 256 --dh 72 --head-stride 80
    python -m paper_2609_29505_gb300.kernel_bench frozen --rows 4096 --d 4096 --caches 8
    python -m paper_2609_29505_gb300.kernel_bench norm --rows 4096 --d 4096
    python -m paper_2609_29505_gb300.kernel_bench trajectory --config dit --budget 0.5 --reps 2
"""
from __future__ import annotations

import argparse
import json
import math

import torch

from . import binding, build

EPI = {"f16": binding.EPI_F16, "f32": binding.EPI_F32, "delta": binding.EPI_DELTA,
       "gated": binding.EPI_GATED, "gelu": binding.EPI_GELU, "rope": binding.EPI_ROPE}


GRAPH = False  # --graph: replay the timed launches from one CUDA graph


def _time(fn, iters, warmup):
    """Average launch time.  Plain: `iters` calls back to back, so a launch shorter than the
    host's per-call work (argument checks, tensor maps, launch) is timed at the host's rate.
    With --graph the calls are captured once into a CUDA graph (on a stream that the warm-up
    calls also used, so the library's per-stream workspace exists before the capture) and
    the replay is timed: device time per launch, as the step programs run them."""
    if not GRAPH:
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(iters):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / iters
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        for _ in range(max(warmup, 1)):
            fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for _ in range(iters):
            fn()
    g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(s):
        e0.record()
        g.replay()
        e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / iters


def case_gemm(a):
    g = torch.Generator(device="cuda").manual_seed(0)
    M, N, K = a.M, a.N, a.K
    rows_b = 2 * N if a.epi == "gated" else N
    A = torch.randn(M, K, device="cuda", generator=g).half()
    B = (torch.randn(rows_b, K, device="cuda", generator=g) / math.sqrt(K)).half()
    epi = binding.sgd_epilogue_args(kind=EPI[a.epi], alpha=1.0)
    keep = []
    if a.epi == "delta":
        h = torch.zeros(M, N, device="cuda")
        cache = torch.empty(M, N, device="cuda", dtype=torch.float16)
        epi.h, epi.ldh = h.data_ptr(), N
        if a.store_cache:
            epi.cache, epi.ld_cache = cache.data_ptr(), N
        keep += [h, cache]
    else:
        out = torch.empty(M, N, device="cuda", dtype=torch.float32 if a.epi == "f32" else torch.float16)
        epi.out, epi.ldo = out.data_ptr(), N
        keep.append(out)
    if a.epi == "rope":
        half = 64
        cos = torch.ones(a.tokens, half, device="cuda")
        sin = torch.zeros(a.tokens, half, device="cuda")
        epi.rope_cos, epi.rope_sin, epi.rope_tokens = cos.data_ptr(), sin.data_ptr(), a.tokens
        epi.d_head, epi.rope_cols = 128, 2 * N // 3
        keep += [cos, sin]
    epi.act = 0
    if a.norm:  # pre-norm folded in: row statistics in a.slots slots (1: finalised by the writer)
        slots = a.slots
        rstat = torch.rand(128, M, device="cuda", generator=g) * (K / slots)
        colsum = torch.randn(rows_b + 512, device="cuda", generator=g)
        colbias = torch.randn(rows_b + 512, device="cuda", generator=g)
        epi.norm = 1 if a.norm == "rms" else 2
        epi.rstat, epi.stat_slots, epi.stat_ld, epi.norm_eps = rstat.data_ptr(), slots, M, 1e-6
        epi.colsum, epi.colbias = colsum.data_ptr(), colbias.data_ptr()
        keep += [rstat, colsum, colbias]
    if a.h16:  # residual writer: fp16 copy of h and row sums
        h16 = torch.empty(M, N, device="cuda", dtype=torch.float16)
        st = torch.empty(128, M, device="cuda")
        fin = torch.empty(128, M, device="cuda")
        cnt = torch.zeros((M + 127) // 128, dtype=torch.int32, device="cuda")
        epi.h16, epi.stat_out, epi.stat_out_ld = h16.data_ptr(), st.data_ptr(), M
        epi.stat_cnt, epi.stat_final = cnt.data_ptr(), fin.data_ptr()
        keep += [h16, st, fin, cnt]
    ms = _time(lambda: binding.sgd_kernel_gemm(A, B, M, N, K, epi, use_simt=a.simt), a.iters, a.warmup)
    flops = 2.0 * M * rows_b * K
    return dict(case="gemm", M=M, N=N, K=K, epi=a.epi, norm=a.norm, h16=a.h16, ms=ms,
                tflops=flops / ms / 1e9)


def case_attention(a):
    B, H, N, dh = a.batch, a.heads, a.tokens, a.dh
    hs = a.head_stride or dh  # input columns per head (80: d_h 72 padded for tcgen05)
    d, w = H * dh, H * hs
    qkv = torch.randn(B * N, 3 * w, device="cuda").half()
    if hs > dh:  # the gaps after every head are zero, as the QKV epilogue leaves them
        qkv.view(B * N, 3 * H, hs)[:, :, dh:] = 0
    o = torch.empty(B * N, d, device="cuda", dtype=torch.float16)
    q, k, v = qkv[:, :w], qkv[:, w:2 * w], qkv[:, 2 * w:]
    ms = _time(lambda: binding.sgd_kernel_attention_hs(q, 3 * w, k, v, 3 * w, hs, o, d, B, N, N, H, dh,
                                                       impl=a.impl), a.iters, a.warmup)
    flops = 4.0 * B * H * N * N * dh
    return dict(case="attention", impl=["tcgen05", "mma_sync", "tcgen05_1tile", "tcgen05_2tile"][a.impl], batch=B, heads=H,
                tokens=N, dh=dh, ms=ms, tflops=flops / ms / 1e9)


def case_frozen(a):
    n = a.rows * a.d
    h = torch.zeros(n, device="cuda")
    caches = [torch.randn(n, device="cuda").half() for _ in range(a.caches)]
    ms = _time(lambda: binding.sgd_kernel_frozen_run(h, caches), a.iters, a.warmup)
    bytes_ = n * (8.0 + 2.0 * a.caches)
    return dict(case="frozen_run", n=n, caches=a.caches, ms=ms, gbs=bytes_ / ms / 1e6)


def case_norm(a):
    h = torch.randn(a.rows, a.d, device="cuda")
    out = torch.empty(a.rows, a.d, device="cuda", dtype=torch.float16)
    g = torch.ones(a.d, device="cuda", dtype=torch.bfloat16)
    ms = _time(lambda: binding.sgd_kernel_norm(h, out, a.rows, a.d, 0, g=g), a.iters, a.warmup)
    return dict(case="norm", rows=a.rows, d=a.d, ms=ms, gbs=6.0 * a.rows * a.d / ms / 1e6)


def case_trajectory(a):
    """Whole trajectories of a synthetic model through sgd_step (its CUDA graphs), timed with
    CUDA events: the launch sequence the step programs run, for launch lists and captures of
    the kernels inside a step."""
    from . import schedule, synth
    cfg = synth.get_config(a.config)
    T = a.T or cfg.T
    w = synth.make_weights(cfg, "cuda")
    inp = synth.make_inputs(cfg, "cuda")
    sched = schedule.build_schedule(cfg, w, T, budget=a.budget)
    model = binding.Denoiser(cfg, w)
    model.set_schedule(T, sched["lifetimes"], sched["groups"])
    if cfg.stem == "embed":
        xs = [synth.token_ids_at(cfg, inp, s, T).cuda() for s in range(1, T + 1)]
    else:
        xs = [inp.z0.cuda()] * T
    if cfg.head == "logits":
        out = torch.empty(cfg.batch, cfg.n_tokens, cfg.d_out, dtype=torch.float16, device="cuda")
    elif cfg.head == "identity":
        out = torch.empty(cfg.batch, cfg.n_tokens, cfg.d, device="cuda")
    else:
        out = torch.empty(cfg.batch, cfg.n_out_tokens, cfg.out_channels, device="cuda")
    cls = None if inp.class_ids is None else inp.class_ids.cuda()
    ctx = None if inp.ctx is None else inp.ctx.cuda()
    times = []
    for _ in range(a.reps):
        model.reset()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for s in range(1, T + 1):
            model.step(xs[s - 1], out, synth.timestep(cfg, s, T), s, class_ids=cls, ctx=ctx)
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    model.check_device()
    model.close()
    ms = min(times) / T
    return dict(case="trajectory", config=a.config, T=T, budget=a.budget, reps=a.reps, ms=ms,
                steps_per_s=1e3 / ms)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("case", choices=["gemm", "attention", "frozen", "norm", "trajectory"])
    ap.add_argument("--config", default="dit", help="trajectory: synthetic model config")
    ap.add_argument("--T", type=int, default=0, help="trajectory: horizon (0: the config's)")
    ap.add_argument("--budget", type=float, default=0.5, help="trajectory: layer-step budget")
    ap.add_argument("--reps", type=int, default=2, help="trajectory: whole trajectories")
    ap.add_argument("--M", type=int, default=4096)
    ap.add_argument("--N", type=int, default=12288)
    ap.add_argument("--K", type=int, default=4096)
    ap.add_argument("--epi", default="f16", choices=list(EPI))
    ap.add_argument("--store-cache", action="store_true")
    ap.add_argument("--norm", default="", choices=["", "rms", "ln"],
                    help="gemm: pre-norm folded into the GEMM (row statistics in 38 slots)")
    ap.add_argument("--slots", type=int, default=1,
                    help="gemm --norm: row-statistic slots the GEMM reads (1: finalised by the writer, "
                         "up to 64: partial sums)")
    ap.add_argument("--h16", action="store_true",
                    help="gemm (delta / f32): also write the fp16 copy of h and the row sums")
    ap.add_argument("--simt", type=int, default=0,
                    help="sgd_kernel_gemm variant: 0 tcgen05 (auto), 1 SIMT, 3 BK 32, "
                         "5 4 epilogue warps, 6 8 warps, 7 128-column tiles, 8 no stream-K, "
                         "9 stream-K forced, 10 128 x 224 tiles, 11 M-fastest tile order, 12 grouped tile order")
    ap.add_argument("--tokens", type=int, default=1024)
    ap.add_argument("--batch", type=int, default=4)
    ap.add_argument("--heads", type=int, default=32)
    ap.add_argument("--dh", type=int, default=128)
    ap.add_argument("--head-stride", type=int, default=0,
                    help="attention: input columns per head (0: d_h; 80 runs d_h 72 on tcgen05)")
    ap.add_argument("--impl", type=int, default=0, help="attention: 0 tcgen05 (auto), 1 mma.sync, 2 tcgen05 one query tile per CTA, "
                         "3 tcgen05 two query tiles per CTA")
    ap.add_argument("--rows", type=int, default=4096)
    ap.add_argument("--d", type=int, default=4096)
    ap.add_argument("--caches", type=int, default=8)
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--graph", action="store_true",
                    help="time the launches replayed from a CUDA graph (device time, no host overhead)")
    a = ap.parse_args()
    global GRAPH
    GRAPH = a.graph
    build.build()
    binding.lib()
    res = {"gemm": case_gemm, "attention": case_attention, "frozen": case_frozen,
           "norm": case_norm, "trajectory": case_trajectory}[a.case](a)
    res["graph"] = a.graph
    res["status"] = binding.sgd_kernel_status()
    print(json.dumps(res))


if __name__ == "__main__":
    main()
