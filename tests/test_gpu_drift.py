"""The causal activation-drift policy (App. B.1) on the GPU against the CPU oracle.

The routing is decided by floating-point drifts, so the comparison is split:
* the GPU's choice at every step is checked exactly against the rule applied to the GPU's
  own drifts (step 1 full, step 2 the m_2 lowest groups, then the m_s largest drifts with
  ties to the lower index), and its active counts against the static schedule's;
* the oracle is teacher-forced on the GPU's states and routing; per step its output must
  match the GPU's within 5e-3 (relative L2) and its drifts the GPU's within the bound
  derived below; where the oracle's own ranking would pick different groups, the groups
  involved must be tied within that bound.

Drift bound: d = ||a - b|| / ||a||.  If the GPU's residual streams a, b carry relative L2
errors up to eps (the per-step output tolerance, 5e-3), then |d_gpu - d_oracle| <=
(||e_a|| + ||e_b||) / ||a|| + d eps / (1 - eps) <= (2 + d) eps (1 + eps).
"""
import numpy as np
import pytest
import torch

from oracle import drift as odr
from oracle import trajectory as otj
from test_gpu_parity import SMALL, STEP_TOL, Case, rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import binding, build
    build.build()
    binding.lib()
    return binding


def drift_tol(d):
    eps = STEP_TOL
    return (2.0 + d) * eps * (1.0 + eps)


def run_gpu(B, c, exec_mode=None):
    """GPU trajectory under the drift policy; the sampler update runs on the host."""
    m = c.model(B)
    m.set_policy(B.POLICY_DRIFT)
    if exec_mode is not None:
        m.set_exec_mode(exec_mode)
    out = c.out_buffer()
    G = m.info()["n_groups"]
    states, outs, masks, drifts = [], [], [], []
    x = None if c.inp.z0 is None else c.inp.z0.numpy().astype(np.float32)
    for s in range(1, c.T + 1):
        if c.cfg.stem == "embed":
            xs = c.ids_at(s)
            states.append(xs.numpy())
            xd = xs.cuda()
        else:
            states.append(x)
            xd = torch.from_numpy(x).cuda()
        m.step(xd, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
        o = out.float().cpu().numpy()
        outs.append(o)
        masks.append(m.active_mask(s))
        drifts.append(m.drift(s))
        if c.cfg.stem != "embed":
            x = (x - o / np.float32(c.T)).astype(np.float32)
    m.check_device()
    info = m.info()
    m.close()
    return dict(states=states, outputs=outs, masks=masks, drift=drifts, G=G, info=info)


def groups_of(c, mask):
    gids = odr.group_order(c.sched["groups"])
    first = [list(c.sched["groups"]).index(g) for g in gids]
    return [i for i, u in enumerate(first) if mask[u]]


_runs = {}


def gpu_run(B, name, budget):
    key = (name, budget)
    if key not in _runs:
        c = Case(name, budget)
        _runs[key] = (c, run_gpu(B, c))
    return _runs[key]


@pytest.mark.parametrize("name", SMALL)
def test_drift_routing_follows_the_rule_on_gpu_drifts(B, name):
    c, g = gpu_run(B, name, 0.5)
    m = odr.static_counts(c.sched["lifetimes"], c.sched["groups"], c.T)
    for s in range(1, c.T + 1):
        picked = groups_of(c, g["masks"][s - 1])
        # the mask is constant over each group
        for u, gid in enumerate(c.sched["groups"]):
            first = list(c.sched["groups"]).index(gid)
            assert g["masks"][s - 1][u] == g["masks"][s - 1][first]
        assert len(picked) == m[s - 1]
        if s == 1:
            assert picked == list(range(g["G"]))
        elif s == 2:
            assert picked == list(range(m[1]))
            assert not np.any(g["drift"][s - 1])
        else:
            assert picked == odr.select(list(g["drift"][s - 1]), m[s - 1])
    info = g["info"]
    assert info["graph_steps"] + info["eager_steps"] == c.T


@pytest.mark.parametrize("name", SMALL)
def test_drift_policy_matches_oracle_teacher_forced(B, name):
    c, g = gpu_run(B, name, 0.5)
    forced = [groups_of(c, mk) for mk in g["masks"]]
    cfg = c.cfg
    ref = odr.run(cfg, c.W, c.sched["lifetimes"], c.sched["groups"], c.T,
                  class_ids=None if c.inp.class_ids is None else c.inp.class_ids.numpy(),
                  ctx=None if c.inp.ctx is None else c.inp.ctx.float().numpy(),
                  ids_at=(lambda s: c.ids_at(s).numpy()) if cfg.stem == "embed" else None,
                  states=None if cfg.stem == "embed" else g["states"], forced=forced)
    errs = [rel(a, b) for a, b in zip(g["outputs"], ref["outputs"])]
    assert max(errs) <= STEP_TOL, f"per-step rel L2 {['%.2e' % e for e in errs]}"
    mcount = odr.static_counts(c.sched["lifetimes"], c.sched["groups"], c.T)
    for s in range(3, c.T + 1):
        dg = np.asarray(g["drift"][s - 1])
        do = np.asarray(ref["drift"][s - 1])
        tol = np.array([drift_tol(v) for v in do])
        assert np.all(np.abs(dg - do) <= tol), (s, np.max(np.abs(dg - do) / tol))
        own = odr.select(list(do), mcount[s - 1])
        if own != forced[s - 1]:
            # both choices valid only if the groups swapped in and out are tied within the bound
            swapped = sorted(set(own) ^ set(forced[s - 1]))
            spread = max(do[swapped]) - min(do[swapped])
            assert spread <= 2 * max(tol[swapped]), (s, swapped, do[swapped])


@pytest.mark.parametrize("name", ["tiny", "llada_small"])
def test_drift_policy_at_full_budget_equals_static(B, name):
    """At a 100% budget every group is active at every step under both policies; the drift
    policy only adds its reductions and cache stores, so the outputs are bit-identical."""
    c = Case(name, 1.0)
    g = run_gpu(B, c)
    m = c.model(B)
    out = c.out_buffer()
    for s in range(1, c.T + 1):
        x = torch.from_numpy(g["states"][s - 1]).cuda()
        m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
        np.testing.assert_array_equal(out.float().cpu().numpy(), g["outputs"][s - 1])
    m.close()


@pytest.mark.parametrize("name", ["dit_small", "llada_small"])
def test_drift_policy_eager_equals_graphs(B, name):
    """Graph replay and op-by-op execution of the drift policy agree bit for bit (routing
    and outputs)."""
    c, g = gpu_run(B, name, 0.5)
    e = run_gpu(B, c, exec_mode=B.EXEC_EAGER)
    assert e["info"]["eager_steps"] == c.T and e["info"]["graph_steps"] == 0
    for a, b in zip(g["masks"], e["masks"]):
        np.testing.assert_array_equal(a, b)
    for a, b in zip(g["outputs"], e["outputs"]):
        np.testing.assert_array_equal(a, b)


def test_drift_policy_state_errors(B):
    c = Case("tiny", 0.5)
    m = c.model(B)
    with pytest.raises(B.SgdError) as err:
        m.drift(1)  # static policy records no drift
    assert err.value.code == B.SGD_ERR_STATE
    m.set_policy(B.POLICY_DRIFT)
    with pytest.raises(B.SgdError) as err:
        m.drift(1)  # not run yet
    assert err.value.code == B.SGD_ERR_STATE
    with pytest.raises(B.SgdError) as err:
        m.set_exec_mode(B.EXEC_PADDED_GRAPH)
    assert err.value.code == B.SGD_ERR_STATE
    m.close()
