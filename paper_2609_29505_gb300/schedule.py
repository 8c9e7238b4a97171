"""Offline schedule construction (Algorithm 1): weights -> scores -> lifetimes.

Host code that runs once per model x horizon x budget; its output (per-unit
lifetimes and atomic groups) is what ``sgd_set_schedule`` consumes.

* spectra: singular values from LAPACK's SVD (float64) for host arrays; for CUDA
  tensors, the eigenvalues of the smaller Gram matrix on the device in fp32 (the
  large synthetic models would take tens of minutes on host cores).
* SCR_eta (Sec. 3.2, Eq. scr-reg) with k = min(d, max(1, floor(0.1 d))),
  g(W) = ||W||_F sqrt(rho(SCR_eta)) (App. G, Eq. app-matrix-score),
  branch scores (Eqs. app-attn-score, app-xattn-score, app-mlp-score),
  unit score = sum over the unit's branches (Eq. app-block-score), normalised by
  max + 1e-12 (Eq. app-score-normalization).
* lifetimes S_l = max{S_min, ceil(T min(1, lam_l / tau))} (Sec. 4.1, Eq. schedule);
  S_min = max(1, floor(0.1 T)) (the paper's S_min = 0.1 T).
* a layer-step budget is met by the tau interval whose lifetimes spend the largest
  number of layer-steps not above floor(budget * G * T + 1e-9): between consecutive
  points tau = T lam_l / j the lifetimes are constant and the spent layer-steps do
  not increase with tau, so the first feasible interval is found by bisection and
  evaluated at its geometric midpoint.

Alternative static rankings (Table tab:cross-ablation) replace the unit score;
they are exposed for latency comparisons at matched budgets.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

ETA = 1e-6


def _is_torch(x) -> bool:
    return type(x).__module__.startswith("torch")


def energies(W):
    """(sigma_i^2 in non-increasing order as float64 NumPy, ||W||_F^2)."""
    if _is_torch(W):
        import torch
        if W.is_cuda:
            prev = torch.backends.cuda.matmul.allow_tf32
            torch.backends.cuda.matmul.allow_tf32 = False
            try:
                A = W.float()
                G = A @ A.T if A.shape[0] <= A.shape[1] else A.T @ A
                ev = torch.linalg.eigvalsh(G)
                fro2 = float((A.double() ** 2).sum())
            finally:
                torch.backends.cuda.matmul.allow_tf32 = prev
            s2 = np.sort(np.clip(ev.double().cpu().numpy(), 0.0, None))[::-1]
            return s2, fro2
        W = W.detach().float().numpy()
    A = np.asarray(W, dtype=np.float64)
    s = np.linalg.svd(A, compute_uv=False)
    return s * s, float(np.einsum("ij,ij->", A, A))


def scr(W, eta: float = ETA) -> float:
    s2, fro2 = energies(W)
    d = s2.size
    k = min(d, max(1, int(0.1 * d)))
    return math.log((s2[:k].sum() + eta * fro2) / (s2[k:].sum() + eta * fro2))


def g_score(W, eta: float = ETA) -> float:
    s2, fro2 = energies(W)
    d = s2.size
    k = min(d, max(1, int(0.1 * d)))
    u = math.log((s2[:k].sum() + eta * fro2) / (s2[k:].sum() + eta * fro2))
    rho = 0.5 * (1.0 + math.tanh(0.5 * u))  # logistic e^u / (1 + e^u)
    return math.sqrt(fro2 * rho)


def _attn_like(gq, gk, gv, go, d_head):
    return go * gv * (1.0 + gq * gk / math.sqrt(d_head))


def _branch_matrices(cfg, weights, b):
    """(kind, [matrices]) for every branch of block b, in graph order."""
    p = f"blocks.{b}."
    d = cfg.d
    out = []
    qkv = weights[p + "w_qkv"]
    out.append(("attn", [qkv[:d], qkv[d:2 * d], qkv[2 * d:], weights[p + "w_o"]]))
    if cfg.block == "xattn":
        kv = weights[p + "wx_kv"]
        out.append(("xattn", [weights[p + "wx_q"], kv[:d], kv[d:], weights[p + "wx_o"]]))
    out.append(("mlp", [weights[p + "w_1"], weights[p + "w_2"]]))
    return out


def branch_scores(cfg, weights, eta: float = ETA, ranking: str = "scr",
                  seed: int = 0) -> np.ndarray:
    """Per-branch raw score in graph order.

    ranking = "scr"   : the paper's SCR/Frobenius score (App. G);
              "frobenius", "spectral", "stable_rank", "frob_stable_rank", "raw_scr":
                        the same branch formulas with g(W) replaced by ||W||_F,
                        ||W||_2, ||W||_F^2/||W||_2^2, their product, or SCR itself;
              "depth"  : later branches score lower; "random": seeded uniform.
    """
    scores: List[float] = []
    idx = 0
    rng = np.random.default_rng(seed)
    n = cfg.n_units
    for b in range(cfg.n_blocks):
        for kind, mats in _branch_matrices(cfg, weights, b):
            if ranking == "depth":
                scores.append(float(n - idx))
            elif ranking == "random":
                scores.append(float(rng.uniform()))
            else:
                gs = [_matrix_stat(W, eta, ranking) for W in mats]
                if kind == "mlp":
                    scores.append(gs[1] * gs[0])
                else:
                    scores.append(_attn_like(*gs, cfg.d_head))
            idx += 1
    return np.asarray(scores, dtype=np.float64)


def _matrix_stat(W, eta, ranking):
    if ranking == "scr":
        return g_score(W, eta)
    s2, fro2 = energies(W)
    if ranking == "frobenius":
        return math.sqrt(fro2)
    if ranking == "spectral":
        return math.sqrt(s2[0])
    if ranking == "stable_rank":
        return fro2 / s2[0]
    if ranking == "frob_stable_rank":
        return math.sqrt(fro2) * fro2 / s2[0]
    if ranking == "raw_scr":
        d = s2.size
        k = min(d, max(1, int(0.1 * d)))
        return math.log((s2[:k].sum() + eta * fro2) / (s2[k:].sum() + eta * fro2))
    raise ValueError(ranking)


def group_scores(branch_q: Sequence[float], groups: Sequence[int]) -> np.ndarray:
    groups = np.asarray(groups)
    q = np.zeros(int(groups.max()) + 1, dtype=np.float64)
    np.add.at(q, groups, np.asarray(branch_q, dtype=np.float64))
    return q


def normalised(q: np.ndarray) -> np.ndarray:
    q = np.asarray(q, dtype=np.float64)
    return q / (q.max() + 1e-12)


def s_min_for(T: int) -> int:
    return max(1, math.floor(0.1 * T))


def lifetimes_for_tau(lam: np.ndarray, T: int, tau: float, s_min: int) -> np.ndarray:
    lam = np.asarray(lam, dtype=np.float64)
    S = np.ceil(T * np.minimum(1.0, lam / tau)).astype(np.int64)
    return np.maximum(S, s_min)


def tau_for_budget(lam: np.ndarray, T: int, budget: float, s_min: int):
    """(tau, lifetimes, feasible) for the largest layer-step count <= the budget."""
    lam = np.asarray(lam, dtype=np.float64)
    cap = math.floor(budget * len(lam) * T + 1e-9)
    pos = lam[lam > 0]
    pts = np.unique((T * pos[:, None] / np.arange(1, T + 1)[None, :]).ravel())
    n = pts.size

    def rep(i):  # representative tau of interval i in 0..n
        if i == 0:
            return pts[0] / 2.0
        if i == n:
            return pts[-1] * 2.0
        return math.sqrt(pts[i - 1] * pts[i])

    def spent(i):
        return int(lifetimes_for_tau(lam, T, rep(i), s_min).sum())

    if spent(n) > cap:
        return math.inf, np.full(len(lam), s_min, dtype=np.int64), False
    lo, hi = 0, n  # first feasible interval lies in [lo, hi]
    while lo < hi:
        mid = (lo + hi) // 2
        if spent(mid) <= cap:
            hi = mid
        else:
            lo = mid + 1
    tau = rep(lo)
    return tau, lifetimes_for_tau(lam, T, tau, s_min), True


def build_schedule(cfg, weights, T: int, budget: Optional[float] = None,
                   tau: Optional[float] = None, granularity: str = "block",
                   s_min: Optional[int] = None, eta: float = ETA, ranking: str = "scr",
                   branch_q: Optional[np.ndarray] = None) -> Dict:
    """Algorithm 1: per-unit lifetimes and atomic groups for ``sgd_set_schedule``.

    Exactly one of ``budget`` (layer-step fraction) and ``tau`` is given.  ``granularity``
    "block" groups the branches of a block (their scores are summed), "branch" schedules
    every branch on its own.  ``branch_q`` reuses precomputed branch scores.
    """
    if (budget is None) == (tau is None):
        raise ValueError("give exactly one of budget and tau")
    nb = len(cfg.branches)
    if granularity == "block":
        groups = np.repeat(np.arange(cfg.n_blocks), nb)
    elif granularity == "branch":
        groups = np.arange(cfg.n_units)
    else:
        raise ValueError(granularity)
    if branch_q is None:
        branch_q = branch_scores(cfg, weights, eta, ranking)
    q = group_scores(branch_q, groups)
    lam = normalised(q)
    s_min = s_min_for(T) if s_min is None else s_min
    feasible = True
    if budget is not None:
        tau, S_g, feasible = tau_for_budget(lam, T, budget, s_min)
    else:
        S_g = lifetimes_for_tau(lam, T, tau, s_min)
    S_u = S_g[groups]
    return dict(lifetimes=S_u.astype(np.int32), groups=groups.astype(np.int32),
                group_lifetimes=S_g, tau=tau, lam=lam, branch_scores=np.asarray(branch_q),
                ratio=float(S_g.sum()) / (len(S_g) * T), feasible=feasible, s_min=s_min, T=T)


# ---------------------------------------------------------------------------
# persistence: a schedule is the only state worth keeping across runs (caches are
# per-trajectory scratch; a resumed run restarts at s = 1)
# ---------------------------------------------------------------------------

SCHEDULE_FORMAT = 1


def weights_digest(weights) -> str:
    """Digest of the weights a schedule was computed from (synth.weights_checksum: exact
    integer checksums of every tensor's raw words, computed where the tensor lives)."""
    from .synth import weights_checksum
    return weights_checksum(weights)


def save_schedule(path: str, sched: Dict, cfg, weights=None, eta: float = ETA,
                  ranking: str = "scr", granularity: str = "block") -> None:
    """Write a schedule from build_schedule (lifetimes, groups, tau, T, S_min, achieved
    ratio) with the knobs that produced it, the model config's name and, when the weights
    are given, their digest."""
    import json
    doc = {
        "format": SCHEDULE_FORMAT, "config": cfg.name, "n_units": int(cfg.n_units),
        "T": int(sched["T"]), "tau": float(sched["tau"]), "eta": float(eta),
        "s_min": int(sched["s_min"]), "ratio": float(sched["ratio"]),
        "feasible": bool(sched["feasible"]), "ranking": ranking, "granularity": granularity,
        "lifetimes": [int(x) for x in sched["lifetimes"]],
        "groups": [int(x) for x in sched["groups"]],
        "weights_digest": weights_digest(weights) if weights is not None else None,
    }
    with open(path, "w") as f:
        json.dump(doc, f, indent=1)


def load_schedule(path: str, cfg=None, weights=None) -> Dict:
    """Read a saved schedule; with `cfg` it must match the model's name and unit count, with
    `weights` their digest (ValueError otherwise).  Returns the fields as build_schedule
    names them (lifetimes and groups as int32 arrays)."""
    import json
    with open(path) as f:
        doc = json.load(f)
    if doc.get("format") != SCHEDULE_FORMAT:
        raise ValueError(f"unknown schedule format {doc.get('format')}")
    if cfg is not None and (doc["config"] != cfg.name or doc["n_units"] != cfg.n_units):
        raise ValueError(f"schedule for {doc['config']} ({doc['n_units']} units), "
                         f"model is {cfg.name} ({cfg.n_units} units)")
    if weights is not None:
        if doc["weights_digest"] is None:
            raise ValueError("schedule was saved without a weights digest")
        if weights_digest(weights) != doc["weights_digest"]:
            raise ValueError("weights differ from the ones the schedule was computed from")
    out = dict(doc)
    out["lifetimes"] = np.asarray(doc["lifetimes"], dtype=np.int32)
    out["groups"] = np.asarray(doc["groups"], dtype=np.int32)
    return out
