"""Pins for the oracle's causal activation-drift policy (App. B.1).

The appendix fixes the drift formula, the top-m_s selection with ties to the lower index,
m_s = the static schedule's active count, a full first step, and frozen units reusing their
last computed update.  These tests check each against hand-computed values, brute force
and special cases that reduce to the static schedule."""
import math

import numpy as np
import pytest

from oracle import denoiser as dn
from oracle import drift as dr
from oracle import trajectory as tj
from paper_2609_29505_gb300 import synth

F32 = np.float32


def _micro(**kw):
    base = dict(name="micro", stem="time_add", block="prenorm", norm="rms", mlp="swiglu",
                head="linear", n_blocks=4, d=32, n_heads=2, d_head=16, d_ff=48, batch=2,
                n_tokens=5, d_in=32, d_out=32, out_channels=32, T=6, seed=7, horizons=[6])
    base.update(kw)
    return synth.ModelConfig(**base)


def _setup(cfg):
    w = dn.to_numpy_weights(synth.make_weights(cfg, "cpu"))
    inp = synth.make_inputs(cfg, "cpu")
    return w, inp.z0.numpy()


def test_lagged_drift_closed_forms():
    n = 50
    a, b = np.full(n, 3.0, F32), np.ones(n, F32)
    assert dr.lagged_drift(a, b) == pytest.approx(2 * math.sqrt(n) / (3 * math.sqrt(n) + 1e-8), rel=1e-15)
    assert dr.lagged_drift(a, a) == 0.0
    # the 1e-8 in the denominator decides when the current input is zero
    assert dr.lagged_drift(np.zeros(4, F32), np.array([3, 4, 0, 0], F32)) == pytest.approx(5 / 1e-8)
    # the norm runs over every element (batch, tokens and width alike)
    x = np.arange(24, dtype=F32).reshape(2, 3, 4)
    y = x.copy()
    y[1, 2, 3] += 2.0
    assert dr.lagged_drift(x, y) == pytest.approx(2.0 / (np.sqrt(np.sum(x.astype(np.float64) ** 2)) + 1e-8))


def test_select_top_m_ties_to_lower_index():
    d = [0.5, 0.9, 0.5, 0.9, 0.1]
    assert dr.select(d, 0) == []
    assert dr.select(d, 1) == [1]
    assert dr.select(d, 2) == [1, 3]
    assert dr.select(d, 3) == [0, 1, 3]
    assert dr.select(d, 4) == [0, 1, 2, 3]
    assert dr.select(d, 5) == [0, 1, 2, 3, 4]
    assert dr.select([0.0] * 6, 3) == [0, 1, 2]


@pytest.mark.parametrize("seed", range(20))
def test_select_brute_force(seed):
    rng = np.random.default_rng(seed)
    G = int(rng.integers(1, 9))
    d = list(rng.integers(0, 4, G).astype(float))  # many ties
    m = int(rng.integers(0, G + 1))
    # brute force: among all m-subsets, the one with the largest drift sum; on a tie, the
    # one whose sorted index list is lexicographically smallest
    import itertools
    best = None
    for sub in itertools.combinations(range(G), m):
        key = (-sum(d[g] for g in sub), list(sub))
        best = key if best is None or key < best else best
    assert dr.select(d, m) == best[1]


def test_static_counts():
    assert dr.static_counts([3, 1, 2], [0, 1, 2], 3) == [3, 2, 1]
    # two-branch groups count once; group ids need not be consecutive numbers
    assert dr.static_counts([2, 2, 3, 3], [5, 5, 7, 7], 3) == [2, 2, 1]
    assert dr.group_order([5, 5, 7, 7, 2]) == [5, 7, 2]


def test_policy_steps_budget_and_first_steps():
    cfg = _micro()
    w, z0 = _setup(cfg)
    T = cfg.T
    S = [6, 6, 3, 3, 2, 2, 4, 4]   # 4 blocks x (attn, mlp), grouped per block
    groups = [0, 0, 1, 1, 2, 2, 3, 3]
    res = dr.run(cfg, w, S, groups, T, z0=z0)
    m = dr.static_counts(S, groups, T)
    assert [len(a) for a in res["active"]] == m
    assert res["active"][0] == [0, 1, 2, 3]        # step 1 full
    assert res["active"][1] == list(range(m[1]))    # step 2: every unit ties
    assert res["drift"][0] is None and res["drift"][1] is None
    for s in range(3, T + 1):
        assert res["active"][s - 1] == dr.select(res["drift"][s - 1], m[s - 1])


def test_policy_equals_static_schedule_when_nothing_is_frozen():
    """With every lifetime = T the policy activates everything at every step and must
    reproduce the static (here: full) trajectory bit for bit."""
    cfg = _micro()
    w, z0 = _setup(cfg)
    S = [cfg.T] * 8
    groups = [0, 0, 1, 1, 2, 2, 3, 3]
    a = dr.run(cfg, w, S, groups, cfg.T, z0=z0)
    b = tj.run(cfg, w, S, cfg.T, z0=z0)
    for x, y in zip(a["outputs"], b["outputs"]):
        np.testing.assert_array_equal(x, y)


def test_drift_values_from_independent_recomputation():
    """The drift the policy uses at step s >= 3 equals the formula applied to the group
    inputs recomputed from scratch: replay steps 1..s-1 with the policy's active sets and
    a fresh cache, tracing each group's first-branch input."""
    cfg = _micro()
    w, z0 = _setup(cfg)
    S = [6, 6, 3, 3, 2, 2, 4, 4]
    groups = [0, 0, 1, 1, 2, 2, 3, 3]
    res = dr.run(cfg, w, S, groups, cfg.T, z0=z0)
    first_unit = [0, 2, 4, 6]
    cache, h_in_steps = {}, []
    for s in range(1, cfg.T + 1):
        act = [groups[u] in res["active"][s - 1] for u in range(8)]
        tr = dn.Trace()
        dn.denoise(cfg, w, res["states"][s - 1], tj.timestep(cfg.T, s), s, S, cache, trace=tr, active_units=act)
        h_in_steps.append({u: hi for (u, _a, hi, _o) in tr.units})
    for s in range(3, cfg.T + 1):
        for g, u in enumerate(first_unit):
            a = h_in_steps[s - 2][u].astype(np.float64)
            b = h_in_steps[s - 3][u].astype(np.float64)
            want = np.linalg.norm(a - b) / (np.linalg.norm(a) + 1e-8)
            assert res["drift"][s - 1][g] == pytest.approx(want, rel=1e-12)


def test_frozen_group_reuses_its_last_computed_update():
    """Whenever a unit is frozen, its contribution (output minus input in the trace) is the
    update it computed at its last active step."""
    cfg = _micro()
    w, z0 = _setup(cfg)
    S = [6, 6, 3, 3, 2, 2, 4, 4]
    groups = [0, 0, 1, 1, 2, 2, 3, 3]
    res = dr.run(cfg, w, S, groups, cfg.T, z0=z0)
    last = {}
    cache = {}
    saw_frozen = False
    for s in range(1, cfg.T + 1):
        act = [groups[u] in res["active"][s - 1] for u in range(8)]
        tr = dn.Trace()
        dn.denoise(cfg, w, res["states"][s - 1], tj.timestep(cfg.T, s), s, S, cache, trace=tr, active_units=act)
        for (u, a, hi, ho) in tr.units:
            if a:
                last[u] = dn.branch(cfg, w, u // 2, cfg.branches[u % 2], hi)
                np.testing.assert_array_equal(ho, (hi + last[u]).astype(F32))
            else:
                saw_frozen = True
                np.testing.assert_array_equal(ho, (hi + last[u]).astype(F32))
    assert saw_frozen


def test_forced_routing_reproduces_the_policy():
    """Teacher-forcing the policy's own choices changes nothing."""
    cfg = _micro()
    w, z0 = _setup(cfg)
    S = [6, 6, 3, 3, 2, 2, 4, 4]
    groups = [0, 0, 1, 1, 2, 2, 3, 3]
    a = dr.run(cfg, w, S, groups, cfg.T, z0=z0)
    b = dr.run(cfg, w, S, groups, cfg.T, z0=z0, forced=a["active"])
    for x, y in zip(a["outputs"], b["outputs"]):
        np.testing.assert_array_equal(x, y)
    assert a["drift"][2:] == b["drift"][2:]


def test_deep_block_input_is_taken_after_the_skip_combine():
    """Reading of App. B.1 for U-ViT: a deep block's drift input is the stream after its long
    skip is combined, W_skip [h ; skip], recomputed here from the traced stream before the
    combine and the pushed shallow-block output."""
    cfg = synth.get_config("uvit_small").with_(n_blocks=3, n_skips=1, d=32, n_heads=2, d_head=16,
                                                d_ff=64, batch=1, n_tokens=6, T=4, n_classes=4)
    w = dn.to_numpy_weights(synth.make_weights(cfg, "cpu"))
    inp = synth.make_inputs(cfg, "cpu")
    S = [4] * cfg.n_units
    groups = list(np.repeat(np.arange(cfg.n_blocks), len(cfg.branches)))
    res = dr.run(cfg, w, S, groups, cfg.T, z0=inp.z0.numpy(), class_ids=inp.class_ids.numpy())
    nb = len(cfg.branches)
    cache, ins = {}, []
    for s in range(1, cfg.T + 1):
        tr = dn.Trace()
        dn.denoise(cfg, w, res["states"][s - 1], tj.timestep(cfg.T, s), s, S, cache,
                   inp.class_ids.numpy(), trace=tr)
        ins.append(tr.units)
    for s in range(3, cfg.T + 1):
        d = []
        for step in (s - 1, s - 2):
            units = ins[step - 1]
            skip = units[nb * 1 - 1][3]          # shallow block 0's output (pushed)
            before = units[nb * 2 - 1][3]        # stream after the middle block
            d.append(dn.skip_combine(w, 0, before, skip))
            np.testing.assert_allclose(units[nb * 2][2], d[-1], rtol=0, atol=0)
        a, b = d[0].astype(np.float64), d[1].astype(np.float64)
        want = np.linalg.norm(a - b) / (np.linalg.norm(a) + 1e-8)
        assert res["drift"][s - 1][2] == pytest.approx(want, rel=1e-12)
