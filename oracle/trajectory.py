"""Sampler loop around the scheduled denoiser (oracle; test infrastructure only).

Sec. 3.1: z_{t-1} = alpha_t z_t - beta_t eps_theta(z_t, t), with evaluations
indexed s = 1..T from the noisiest state.  Reading: alpha = 1, beta = 1/T and
t_s = 1000 (T - s + 1) / T.  Token models (LLaDA) take their ids at step s from a
seeded reveal sequence that does not depend on the outputs, so the state at
every step is an input (see ``ids_at``).
"""
from __future__ import annotations

import time
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

from . import denoiser

F32 = np.float32


def timestep(T: int, s: int) -> float:
    return 1000.0 * (T - s + 1) / T


def run(cfg, weights, S_units: Sequence[int], T: int, z0=None, class_ids=None, ctx=None,
        ids_at: Optional[Callable[[int], np.ndarray]] = None, steps: Optional[int] = None,
        states: Optional[List[np.ndarray]] = None) -> Dict:
    """Closed-loop scheduled trajectory.

    Returns dict(states=[z_1..z_{T+1}], outputs=[eps_1..eps_T]).  For token models the
    states are the id tensors from ``ids_at`` and nothing is integrated.  ``steps``
    truncates the trajectory.  If ``states`` is given, step s is evaluated on
    ``states[s-1]`` (teacher forcing) instead of the integrated state.
    """
    cache: Dict[int, np.ndarray] = {}
    outs: List[np.ndarray] = []
    zs: List[np.ndarray] = []
    z = None if z0 is None else np.asarray(z0, dtype=F32)
    n = T if steps is None else steps
    for s in range(1, n + 1):
        t = timestep(T, s)
        if ids_at is not None:
            x = np.asarray(ids_at(s))
        elif states is not None:
            x = np.asarray(states[s - 1], dtype=F32)
        else:
            x = z
        zs.append(x)
        eps = denoiser.denoise(cfg, weights, x, t, s, S_units, cache, class_ids, ctx)
        outs.append(eps)
        if ids_at is None:
            z = (x - eps / F32(T)).astype(F32)
    if ids_at is None:
        zs.append(z)
    return dict(states=zs, outputs=outs)


def time_steps(cfg, weights, S_units, T, step_list, state_fn, class_ids=None, ctx=None):
    """Wall time of the oracle at the given steps (caches built by running the steps
    before each one untimed would cost as much; instead every unit is treated as
    having a cache filled with zeros, which does not change the work done)."""
    cache = {u: 0.0 for u in range(len(S_units))}
    times = []
    for s in step_list:
        t0 = time.perf_counter()
        denoiser.denoise(cfg, weights, state_fn(s), timestep(T, s), s, S_units, cache,
                         class_ids, ctx)
        times.append(time.perf_counter() - t0)
    return times
