"""Parity at the full workload sizes, in the launch configuration bench.py times.

The GPU runs the whole batch of each full-size synthetic model (its graphs are the
ones the benchmark replays); the CPU oracle evaluates batch row 0 alone, which is
exact because every operation of these models is per sample.  Active sets are
compared bit for bit, eps / logits of row 0 per step (teacher forced, relative L2
<= 5e-3) and, for the continuous models, the closed-loop final state of row 0
(relative L2 <= 1e-2).  The LLaDA-shaped model uses its 10-step horizon.
"""
import numpy as np
import pytest
import torch

from oracle import denoiser as odn
from oracle import spectral as osp
from oracle import trajectory as otj
from paper_2609_29505_gb300 import schedule, synth

pytestmark = pytest.mark.gpu

STEP_TOL = 5e-3
FINAL_TOL = 1e-2
# (config, horizon, budget)
CASES = [("tiny", 10, 0.5), ("dit", 50, 0.5), ("uvit", 50, 0.5), ("sdxl", 30, 0.5),
         ("llada", 10, 0.5)]


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import binding, build
    build.build()
    binding.lib()
    return binding


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


@pytest.mark.parametrize("name,T,budget", CASES, ids=[c[0] for c in CASES])
def test_full_size_row0(B, name, T, budget):
    cfg = synth.get_config(name)
    dev = torch.device("cuda")
    w = synth.make_weights(cfg, dev)
    inp = synth.make_inputs(cfg, dev)
    sched = schedule.build_schedule(cfg, w, T, budget=budget)
    S = sched["lifetimes"]
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

    if cfg.head == "logits":
        out = torch.empty(cfg.batch, cfg.n_tokens, cfg.d_out, dtype=torch.float16, device=dev)
    elif cfg.head == "identity":
        out = torch.empty(cfg.batch, cfg.n_tokens, cfg.d, device=dev)
    else:
        out = torch.empty(cfg.batch, cfg.n_out_tokens, cfg.out_channels, device=dev)

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
