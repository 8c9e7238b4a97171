"""Parity at the full workload sizes, in the launch configuration bench.py times.

* Schedules: for every full-size model, horizon and budget (100 / 50 / 33%), the
  product's lifetimes (schedule.build_schedule, device spectra) equal the oracle's
  (oracle.spectral, float64 host spectra; stored in tests/golden/full_size_schedules.json
  for these exact weights, else computed here) as integers, and the library's active
  sets equal the oracle's A_s bit for bit.
* Trajectories: the GPU runs the whole batch of each model (its graphs are the ones the
  benchmark replays); the CPU oracle evaluates batch row 0 alone, which is exact because
  every operation of these models is per sample.  eps / logits of row 0 are compared per
  step (teacher forced, relative L2 <= 5e-3) and, for the continuous models, the
  closed-loop final state of row 0 (relative L2 <= 1e-2).
* The LLaDA-shaped model at its benchmarked horizon (T = 64, 50%): the oracle evaluates
  only the steps the comparison needs -- the last step of every active pattern (the step
  s = S_l at which the pattern's units store their updates) and the first step of the two
  last patterns, plus steps 1 and T -- on sampled token rows of the logits.  Skipping the
  other steps leaves the oracle's caches unchanged: a step that is no unit's S_l only
  refreshes caches that a later evaluated step (that unit's S_l) overwrites.
"""
import os
import sys

import numpy as np
import pytest
import torch

from oracle import denoiser as odn
from oracle import spectral as osp
from oracle import trajectory as otj
from paper_2609_29505_gb300 import schedule, synth

sys.path.insert(0, os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden"))
import full_size_schedules as golden  # noqa: E402

pytestmark = pytest.mark.gpu

STEP_TOL = 5e-3
FINAL_TOL = 1e-2
# (config, horizon, budget)
CASES = [("tiny", 10, 0.5), ("dit", 50, 0.5), ("uvit", 50, 0.5), ("sdxl", 30, 0.5),
         ("llada", 10, 0.5), ("dit", 50, 1.0), ("dit", 50, 0.33), ("sdxl", 30, 1.0),
         ("sdxl", 30, 0.33)]
SCHEDULE_MODELS = ["tiny", "dit", "uvit", "sdxl", "llada"]


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import binding, build
    build.build()
    binding.lib()
    return binding


_weights = {}


def weights(name):
    """Full-size weights of one model on the device (the last model's are kept)."""
    if name not in _weights:
        _weights.clear()
        torch.cuda.empty_cache()
        cfg = synth.get_config(name)
        _weights[name] = synth.make_weights(cfg, torch.device("cuda"))
    return _weights[name]


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def oracle_lifetimes(cfg, w, T, budget):
    S, _ = golden.oracle_lifetimes(cfg, w, T, budget)
    return S


@pytest.mark.parametrize("name", SCHEDULE_MODELS)
def test_full_size_schedules_equal_oracle(B, name):
    """Algorithm 1 at full size: product lifetimes == oracle lifetimes (integers) at every
    horizon of the model and every budget, and the library's per-step active sets ==
    the oracle's A_s."""
    cfg = synth.get_config(name)
    w = weights(name)
    bq = None
    for T in cfg.horizons:
        for budget in synth.BUDGETS:
            sched = schedule.build_schedule(cfg, w, T, budget=budget, branch_q=bq)
            bq = sched["branch_scores"]
            S = oracle_lifetimes(cfg, w, T, budget)
            np.testing.assert_array_equal(sched["lifetimes"], S, err_msg=f"T={T} budget={budget}")
            if budget == 0.5:
                model = B.Denoiser(cfg, w)
                model.set_schedule(T, S, sched["groups"])
                masks = osp.active_sets(S, T)
                for s in range(1, T + 1):
                    np.testing.assert_array_equal(model.active_mask(s), masks[s - 1])
                model.close()


def out_buffer(cfg, dev):
    if cfg.head == "logits":
        return torch.empty(cfg.batch, cfg.n_tokens, cfg.d_out, dtype=torch.float16, device=dev)
    if cfg.head == "identity":
        return torch.empty(cfg.batch, cfg.n_tokens, cfg.d, device=dev)
    return torch.empty(cfg.batch, cfg.n_out_tokens, cfg.out_channels, device=dev)


@pytest.mark.parametrize("name,T,budget", CASES, ids=[f"{c[0]}-T{c[1]}-{c[2]:g}" for c in CASES])
def test_full_size_row0(B, name, T, budget):
    cfg = synth.get_config(name)
    dev = torch.device("cuda")
    w = weights(name)
    inp = synth.make_inputs(cfg, dev)
    sched = schedule.build_schedule(cfg, w, T, budget=budget)
    S = oracle_lifetimes(cfg, w, T, budget)
    np.testing.assert_array_equal(sched["lifetimes"], S)
    model = B.Denoiser(cfg, w)
    model.set_schedule(T, S, sched["groups"])
    masks = osp.active_sets(S, T)
    for s in range(1, T + 1):
        np.testing.assert_array_equal(model.active_mask(s), masks[s - 1])

    # oracle on batch row 0
    ocfg = cfg.with_(batch=1)
    W = {k: v.float().cpu().numpy() for k, v in w.items()}
    cls = None if inp.class_ids is None else inp.class_ids.to(dev)
    ctx = None if inp.ctx is None else inp.ctx.to(dev)
    cls0 = None if inp.class_ids is None else inp.class_ids[:1].cpu().numpy()
    ctx0 = None if inp.ctx is None else inp.ctx[:1].float().cpu().numpy()
    token = cfg.stem == "embed"
    ids_at = (lambda s: synth.token_ids_at(cfg, inp, s, T)) if token else None
    ref = otj.run(ocfg, W, S, T, z0=None if token else inp.z0[:1].cpu().numpy(),
                  class_ids=cls0, ctx=ctx0,
                  ids_at=(lambda s: ids_at(s)[:1].cpu().numpy()) if token else None)
    del W

    out = out_buffer(cfg, dev)
    # teacher forced: row 0 gets the oracle's state, the other rows keep the seeded input
    errs = []
    for s in range(1, T + 1):
        if token:
            x = ids_at(s).to(dev)
        else:
            x = inp.z0.clone()
            x[0] = torch.from_numpy(ref["states"][s - 1][0]).to(dev)
        model.step(x, out, otj.timestep(T, s), s, class_ids=cls, ctx=ctx)
        errs.append(rel(out[0].float().cpu().numpy(), ref["outputs"][s - 1][0]))
    model.check_device()
    assert max(errs) <= STEP_TOL, f"per-step rel L2 {['%.2e' % e for e in errs]}"

    if cfg.norm in ("rms", "ln") and budget == 0.5:  # the same with the pre-norms folded in
        fm = B.Denoiser(cfg, w, flags=B.FLAG_FOLD_NORM)
        fm.set_schedule(T, S, sched["groups"])
        ferrs = []
        for s in range(1, T + 1):
            if token:
                x = ids_at(s).to(dev)
            else:
                x = inp.z0.clone()
                x[0] = torch.from_numpy(ref["states"][s - 1][0]).to(dev)
            fm.step(x, out, otj.timestep(T, s), s, class_ids=cls, ctx=ctx)
            ferrs.append(rel(out[0].float().cpu().numpy(), ref["outputs"][s - 1][0]))
        fm.check_device()
        fm.close()
        assert max(ferrs) <= STEP_TOL, f"folded norms: per-step rel L2 {['%.2e' % e for e in ferrs]}"

    if not token:  # closed loop on the GPU's own states
        z = inp.z0.clone()
        model.reset()
        for s in range(1, T + 1):
            model.step(z, out, otj.timestep(T, s), s, class_ids=cls, ctx=ctx)
            B.sgd_sampler_update(z, out, 1.0, 1.0 / T)
        torch.cuda.synchronize()
        assert rel(z[0].cpu().numpy(), ref["states"][-1][0]) <= FINAL_TOL
        assert rel(out[0].cpu().numpy(), ref["outputs"][-1][0]) <= FINAL_TOL
    model.close()


def test_full_size_llada_T64_budget50(B):
    """The benchmarked workload: LLaDA-8B-shaped, batch 4 x 1024, T = 64, 50% budget.
    Every active pattern is checked at its last step (and the last two patterns also at
    their first step), on 64 seeded token rows of batch row 0's logits."""
    name, T, budget = "llada", 64, 0.5
    cfg = synth.get_config(name)
    dev = torch.device("cuda")
    w = weights(name)
    inp = synth.make_inputs(cfg, dev)
    sched = schedule.build_schedule(cfg, w, T, budget=budget)
    S = oracle_lifetimes(cfg, w, T, budget)
    np.testing.assert_array_equal(sched["lifetimes"], S)
    lifetimes = sorted({int(x) for x in S if x < T})
    checks = sorted({1, T, *lifetimes, *[x + 1 for x in lifetimes[-2:]]})
    evaluated = sorted(set(checks) | set(lifetimes))
    rows = np.sort(np.random.default_rng(7).choice(cfg.n_tokens, 64, replace=False))

    # GPU: every step of the trajectory, in order (its caches need them)
    model = B.Denoiser(cfg, w)
    model.set_schedule(T, S, sched["groups"])
    out = out_buffer(cfg, dev)
    got = {}
    for s in range(1, T + 1):
        model.step(synth.token_ids_at(cfg, inp, s, T).to(dev), out, otj.timestep(T, s), s)
        if s in checks:
            got[s] = out[0, torch.from_numpy(rows).to(dev)].float().cpu().numpy()
    model.check_device()
    model.close()

    # oracle: row 0, only the evaluated steps, head on the sampled rows
    ocfg = cfg.with_(batch=1)
    W = {k: v.float().cpu().numpy() for k, v in w.items()}
    cache = {}
    errs = {}
    for s in evaluated:
        ids = synth.token_ids_at(cfg, inp, s, T)[:1].cpu().numpy()
        h, c = odn.denoise(ocfg, W, ids, otj.timestep(T, s), s, S, cache, with_head=False)
        if s in checks:
            want = odn.head(ocfg, W, h[:, rows], c)[0]
            errs[s] = rel(got[s], want)
    del W
    assert max(errs.values()) <= STEP_TOL, f"per-step rel L2 {errs}"
