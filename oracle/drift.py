"""Causal activation-drift policy (App. B.1, "Causal activation drift"): the input-aware
baseline that the static schedule is compared with (Table tab:input-aware).

Test infrastructure only: used by tests/, never by the product path.

After step s-1 the policy records, for every scheduled unit l, the lagged drift of the
unit's input h_{l-1} (the residual stream entering the unit),

    d_{l,s-1} = ||h_{l-1,s-1} - h_{l-1,s-2}||_2 / (||h_{l-1,s-1}||_2 + 1e-8),

and at step s activates exactly the m_s units with the largest lagged drift, m_s being the
static schedule's active count at step s; ties go to the lower unit index; step 1 is full.
A frozen unit adds the update it computed at its last active step.

Readings (the appendix does not say):
  * a scheduled unit is an atomic group of branches (a block by default); its input is
    the residual stream entering the group's first branch, after any U-ViT skip-combine;
  * the batch shares one active set, so the norms run over the whole [B, N, d] tensor;
  * at step 2 no lagged drift exists yet (it needs inputs from two earlier steps), so every
    unit ties and the m_2 lowest-indexed units are active.
Drift values are computed in float64 from the float32 residual stream.
"""
from __future__ import annotations

from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

from . import denoiser
from .trajectory import timestep

F32 = np.float32


def lagged_drift(h_now: np.ndarray, h_prev: np.ndarray) -> float:
    """d = ||h_now - h_prev||_2 / (||h_now||_2 + 1e-8) over all elements (App. B.1)."""
    a = np.asarray(h_now, dtype=np.float64).ravel()
    b = np.asarray(h_prev, dtype=np.float64).ravel()
    return float(np.sqrt(np.sum((a - b) ** 2)) / (np.sqrt(np.sum(a * a)) + 1e-8))


def select(drift: Sequence[float], m: int) -> List[int]:
    """Indices of the m largest drifts, ties to the lower index; returned in ascending order."""
    order = sorted(range(len(drift)), key=lambda g: (-drift[g], g))
    return sorted(order[:m])


def group_order(groups: Sequence[int]) -> List[int]:
    """Distinct group ids in the order of their first unit (the unit index of a group)."""
    seen: List[int] = []
    for g in groups:
        if g not in seen:
            seen.append(g)
    return seen


def static_counts(S_units: Sequence[int], groups: Sequence[int], T: int) -> List[int]:
    """m_s for s = 1..T: how many groups the static schedule runs at step s (s <= S_g)."""
    ids = group_order(groups)
    life = {g: S_units[list(groups).index(g)] for g in ids}
    return [sum(1 for g in ids if life[g] >= s) for s in range(1, T + 1)]


def run(cfg, weights, S_units: Sequence[int], groups: Sequence[int], T: int, z0=None,
        class_ids=None, ctx=None, ids_at: Optional[Callable[[int], np.ndarray]] = None,
        steps: Optional[int] = None, states: Optional[List[np.ndarray]] = None,
        forced: Optional[List[Sequence[int]]] = None) -> Dict:
    """Trajectory under the drift policy (same sampler as trajectory.run).

    Returns dict(states, outputs, active=[active group indices per step],
    drift=[per step s >= 3: the lagged drifts d_{., s-1} the selection used]).
    ``forced``, when given, makes step s run the groups forced[s-1] instead of the policy's
    choice (teacher forcing of the routing; the drifts are still computed and returned).
    """
    ids = group_order(groups)
    G = len(ids)
    units_of = [[u for u in range(len(groups)) if groups[u] == g] for g in ids]
    m = static_counts(S_units, groups, T)
    cache: Dict[int, np.ndarray] = {}
    outs: List[np.ndarray] = []
    zs: List[np.ndarray] = []
    chosen: List[List[int]] = []
    drifts: List[Optional[List[float]]] = []
    inputs: List[List[np.ndarray]] = []  # per step: the input of every group
    z = None if z0 is None else np.asarray(z0, dtype=F32)
    n = T if steps is None else steps
    for s in range(1, n + 1):
        if s == 1:
            d = None
            pick = list(range(G))
        elif s == 2:
            d = None
            pick = list(range(m[s - 1]))
        else:
            d = [lagged_drift(inputs[-1][g], inputs[-2][g]) for g in range(G)]
            pick = select(d, m[s - 1])
        if forced is not None:
            pick = sorted(forced[s - 1])
        chosen.append(pick)
        drifts.append(d)
        act = [False] * len(groups)
        for g in pick:
            for u in units_of[g]:
                act[u] = True
        t = timestep(T, s)
        if ids_at is not None:
            x = np.asarray(ids_at(s))
        elif states is not None:
            x = np.asarray(states[s - 1], dtype=F32)
        else:
            x = z
        zs.append(x)
        tr = denoiser.Trace()
        eps = denoiser.denoise(cfg, weights, x, t, s, S_units, cache, class_ids, ctx, trace=tr,
                               active_units=act)
        h_in = {u: hi for (u, _a, hi, _ho) in tr.units}
        inputs.append([h_in[units_of[g][0]] for g in range(G)])
        if len(inputs) > 2:
            inputs.pop(0)
        outs.append(eps)
        if ids_at is None:
            z = (x - eps / F32(T)).astype(F32)
    if ids_at is None:
        zs.append(z)
    return dict(states=zs, outputs=outs, active=chosen, drift=drifts)
