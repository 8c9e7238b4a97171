"""Weight-only scores and static lifetimes (oracle; test infrastructure only).

Every function follows one passage of the paper:

* ``singular_energies`` / ``scr_eta``  — Sec. 3.2, Definition of the regularised
  Spectral Concentration Ratio (Eq. scr-reg).
* ``matrix_score``                      — App. G, Eq. app-matrix-score
  (g(W) = ||W||_F sqrt(rho(SCR_eta(W))), rho the logistic function); the same
  quantity is gamma_j in Sec. 3.3.
* ``attn_score`` / ``xattn_score`` / ``mlp_score`` — App. G, Eqs. app-attn-score,
  app-xattn-score, app-mlp-score.
* ``unit_scores``                       — App. G, Eq. app-block-score (sum over the
  scheduled unit's submodules).
* ``normalise``                         — App. G, Eq. app-score-normalization
  (epsilon = 1e-12).
* ``lifetimes``                         — Sec. 4.1, Eq. schedule.
* ``tau_for_budget``                    — reading: the paper sets tau and reports the
  resulting layer-step ratio; a requested budget is met by the tau interval whose
  ratio is the largest not above the budget.
* ``active_sets``                       — Sec. 3.1 / Algorithm 2: unit l is evaluated
  at step s iff s <= S_l.
* ``matrix_statistic`` / ``ranked_branch_scores`` — the alternative static rankings of
  Table tab:cross-ablation (random, depth-only, Frobenius norm, spectral norm, stable
  rank, Frobenius x stable rank, raw SCR).  Reading: each replaces g(W) in the branch
  formulas of App. G by its own per-matrix statistic, larger scores giving longer
  lifetimes; depth-only scores a branch by its distance from the output (earlier
  branches live longer); random takes the draws it is given.
"""
from __future__ import annotations

import math
from typing import Dict, List, Sequence, Tuple

import numpy as np

ETA = 1e-6            # eta > 0 (Sec. 3.2); the paper does not print a value
NORM_EPS = 1e-12      # epsilon of Eq. app-score-normalization


def singular_energies(W) -> np.ndarray:
    """sigma_i^2, i = 1..d, d = min(m, n), in non-increasing order.

    Computed as the eigenvalues of the smaller Gram matrix in float64 (clamped at
    zero: the Gram matrix is positive semidefinite).
    """
    A = np.asarray(W, dtype=np.float64)
    m, n = A.shape
    gram = A @ A.T if m <= n else A.T @ A
    ev = np.linalg.eigvalsh(gram)
    ev = np.clip(ev, 0.0, None)
    return np.sort(ev)[::-1]


def top_k(d: int) -> int:
    """k = min(d, max(1, floor(0.1 d)))  (Sec. 3.2)."""
    return min(d, max(1, int(math.floor(0.1 * d))))


def frobenius_sq(W) -> float:
    """||W||_F^2 as the sum of squared entries."""
    A = np.asarray(W, dtype=np.float64)
    return float(np.sum(A * A))


def scr_eta(W, eta: float = ETA) -> float:
    """Regularised SCR (Eq. scr-reg):
    log( (sum_{i<=k} sigma_i^2 + eta ||W||_F^2) / (sum_{i>k} sigma_i^2 + eta ||W||_F^2) )."""
    s2 = singular_energies(W)
    k = top_k(s2.size)
    f2 = frobenius_sq(W)
    lead = float(np.sum(s2[:k]))
    tail = float(np.sum(s2[k:]))
    return math.log((lead + eta * f2) / (tail + eta * f2))


def logistic(u: float) -> float:
    """rho(u) = e^u / (1 + e^u)  (Lemma lem:sandwich, Eq. app-matrix-score)."""
    if u >= 0:
        return 1.0 / (1.0 + math.exp(-u))
    e = math.exp(u)
    return e / (1.0 + e)


def matrix_score(W, eta: float = ETA) -> float:
    """g(W) = ||W||_F sqrt(rho(SCR_eta(W)))  (Eq. app-matrix-score)."""
    return math.sqrt(frobenius_sq(W)) * math.sqrt(logistic(scr_eta(W, eta)))


def attn_score(Wq, Wk, Wv, Wo, d_head: int, eta: float = ETA) -> float:
    """q_attn = g(W_O) g(W_V) [1 + g(W_Q) g(W_K) / sqrt(d_h)]  (Eq. app-attn-score)."""
    gq, gk, gv, go = (matrix_score(w, eta) for w in (Wq, Wk, Wv, Wo))
    return go * gv * (1.0 + gq * gk / math.sqrt(d_head))


def xattn_score(Wq, Wk, Wv, Wo, d_head: int, eta: float = ETA) -> float:
    """Cross-attention: the same form, W_K and W_V act on the conditioning sequence
    (Eq. app-xattn-score)."""
    return attn_score(Wq, Wk, Wv, Wo, d_head, eta)


def mlp_score(W1, W2, eta: float = ETA) -> float:
    """q_mlp = g(W_2) g(W_1)  (Eq. app-mlp-score)."""
    return matrix_score(W2, eta) * matrix_score(W1, eta)


def branch_scores(cfg, weights: Dict[str, np.ndarray], eta: float = ETA) -> List[float]:
    """Score of every residual branch, in graph order (attn[, xattn], mlp per block).

    Scored matrices (reading): the attention projections (W_Q, W_K, W_V are the three
    d x d row blocks of the stacked QKV weight), the cross-attention projections (K and
    V are the two row blocks of the context projection), and the MLP input/output
    projections (for gated MLPs W_1 is the stacked [gate; up] or [a; b] matrix).
    """
    d = cfg.d
    out: List[float] = []
    for b in range(cfg.n_blocks):
        p = f"blocks.{b}."
        wqkv = weights[p + "w_qkv"]
        out.append(attn_score(wqkv[:d], wqkv[d:2 * d], wqkv[2 * d:], weights[p + "w_o"],
                              cfg.d_head, eta))
        if cfg.block == "xattn":
            wkv = weights[p + "wx_kv"]
            out.append(xattn_score(weights[p + "wx_q"], wkv[:d], wkv[d:], weights[p + "wx_o"],
                                   cfg.d_head, eta))
        out.append(mlp_score(weights[p + "w_1"], weights[p + "w_2"], eta))
    return out


RANKINGS = ("scr", "frobenius", "spectral", "stable_rank", "frob_stable_rank", "raw_scr",
            "depth", "random")


def matrix_statistic(W, ranking: str, eta: float = ETA) -> float:
    """Per-matrix score of one static ranking (Table tab:cross-ablation):
    scr -> g(W); frobenius -> ||W||_F; spectral -> ||W||_2 = sigma_1;
    stable_rank -> ||W||_F^2 / ||W||_2^2; frob_stable_rank -> ||W||_F times the stable
    rank; raw_scr -> SCR_eta(W) (Eq. scr-reg)."""
    if ranking == "scr":
        return matrix_score(W, eta)
    if ranking == "raw_scr":
        return scr_eta(W, eta)
    f2 = frobenius_sq(W)
    if ranking == "frobenius":
        return math.sqrt(f2)
    top = float(singular_energies(W)[0])
    if ranking == "spectral":
        return math.sqrt(top)
    if ranking == "stable_rank":
        return f2 / top
    if ranking == "frob_stable_rank":
        return math.sqrt(f2) * (f2 / top)
    raise ValueError(ranking)


def ranked_branch_scores(cfg, weights, ranking: str, eta: float = ETA,
                         draws: Sequence[float] = None) -> List[float]:
    """Branch scores of one static ranking, in graph order.  Matrix rankings use the
    branch formulas of App. G (Eqs. app-attn-score, app-xattn-score, app-mlp-score) with
    matrix_statistic in place of g; depth-only gives branch u of U the score U - u;
    random returns ``draws`` (one per branch, drawn by the caller)."""
    n = cfg.n_units
    if ranking == "depth":
        return [float(n - u) for u in range(n)]
    if ranking == "random":
        if draws is None or len(draws) != n:
            raise ValueError("the random ranking takes one draw per branch")
        return [float(x) for x in draws]
    st = lambda W: matrix_statistic(W, ranking, eta)
    d = cfg.d
    out: List[float] = []
    for b in range(cfg.n_blocks):
        p = f"blocks.{b}."
        wqkv = weights[p + "w_qkv"]
        gq, gk, gv, go = st(wqkv[:d]), st(wqkv[d:2 * d]), st(wqkv[2 * d:]), st(weights[p + "w_o"])
        out.append(go * gv * (1.0 + gq * gk / math.sqrt(cfg.d_head)))
        if cfg.block == "xattn":
            wkv = weights[p + "wx_kv"]
            gq, gk, gv, go = st(weights[p + "wx_q"]), st(wkv[:d]), st(wkv[d:]), st(weights[p + "wx_o"])
            out.append(go * gv * (1.0 + gq * gk / math.sqrt(cfg.d_head)))
        out.append(st(weights[p + "w_2"]) * st(weights[p + "w_1"]))
    return out


def unit_scores(branch_q: Sequence[float], group_of_unit: Sequence[int]) -> np.ndarray:
    """Raw unit score q~_l = sum of the scores of the unit's submodules
    (Eq. app-block-score).  Groups are numbered 0..G-1 in order of appearance."""
    n_groups = max(group_of_unit) + 1
    q = np.zeros(n_groups, dtype=np.float64)
    for u, g in enumerate(group_of_unit):
        q[g] += branch_q[u]
    return q


def normalise(q: np.ndarray, eps: float = NORM_EPS) -> np.ndarray:
    """Lambda^_l = q~_l / (max_j q~_j + eps)  (Eq. app-score-normalization)."""
    q = np.asarray(q, dtype=np.float64)
    return q / (np.max(q) + eps)


def min_lifetime(T: int) -> int:
    """S_min = 0.1 T (Sec. 5.2 default) read as max(1, floor(0.1 T))."""
    return max(1, int(math.floor(0.1 * T)))


def lifetimes(lam: np.ndarray, T: int, tau: float, s_min: int) -> np.ndarray:
    """S_l = max{S_min, ceil(T min(1, Lambda^_l / tau))}  (Eq. schedule)."""
    out = np.empty(len(lam), dtype=np.int64)
    for l, x in enumerate(lam):
        out[l] = max(s_min, int(math.ceil(T * min(1.0, float(x) / tau))))
    return out


def budget_cap(budget: float, n_groups: int, T: int) -> int:
    """Largest admissible sum of lifetimes: floor(budget * G * T) (1e-9 guards the
    representation error of decimal budgets such as 0.33)."""
    return int(math.floor(budget * n_groups * T + 1e-9))


def tau_for_budget(lam: np.ndarray, T: int, budget: float, s_min: int
                   ) -> Tuple[float, np.ndarray, bool]:
    """Scale tau whose lifetimes use the largest layer-step ratio not above ``budget``.

    S_l(tau) changes only where T Lambda^_l / tau crosses an integer j, i.e. at
    tau = T Lambda^_l / j.  Between consecutive such points the lifetimes are constant;
    each open interval is evaluated at its geometric midpoint (below the smallest
    point: half of it; above the largest: twice it).  Returns (tau, lifetimes,
    feasible); when even the all-S_min schedule exceeds the budget it is returned
    with feasible = False.
    """
    lam = np.asarray(lam, dtype=np.float64)
    G = len(lam)
    cap = budget_cap(budget, G, T)
    points = sorted({T * float(x) / j for x in lam if x > 0 for j in range(1, T + 1)})
    reps = [points[0] / 2.0]
    for a, b in zip(points[:-1], points[1:]):
        reps.append(math.sqrt(a * b))
    reps.append(points[-1] * 2.0)
    best = None
    for tau in reps:
        S = lifetimes(lam, T, tau, s_min)
        total = int(S.sum())
        if total <= cap and (best is None or total > best[2]):
            best = (tau, S, total)
    if best is None:
        S = np.full(G, s_min, dtype=np.int64)
        return math.inf, S, False
    return best[0], best[1], True


def layer_step_ratio(S: np.ndarray, T: int) -> float:
    """Achieved budget sum_l S_l / (L T)."""
    return float(np.sum(S)) / (len(S) * T)


def active_sets(S_units: Sequence[int], T: int) -> np.ndarray:
    """uint8 [T, U]: entry (s-1, u) is 1 iff unit u is evaluated at step s (s <= S_u)."""
    S = np.asarray(S_units)
    mask = np.zeros((T, len(S)), dtype=np.uint8)
    for s in range(1, T + 1):
        for u in range(len(S)):
            mask[s - 1, u] = 1 if s <= S[u] else 0
    return mask


def schedule(cfg, weights: Dict[str, np.ndarray], T: int, budget: float,
             group_of_unit: Sequence[int], eta: float = ETA, branch_q=None) -> Dict:
    """Algorithm 1 end to end: scores -> normalised scores -> tau -> per-unit lifetimes.
    ``branch_q``: the branch scores of these weights, when already computed by
    ``branch_scores`` (the weights are then not read)."""
    bq = branch_scores(cfg, weights, eta) if branch_q is None else [float(x) for x in branch_q]
    q = unit_scores(bq, group_of_unit)
    lam = normalise(q)
    s_min = min_lifetime(T)
    tau, S_groups, feasible = tau_for_budget(lam, T, budget, s_min)
    S_units = np.array([S_groups[g] for g in group_of_unit], dtype=np.int64)
    return dict(branch_scores=np.array(bq), unit_scores=q, lam=lam, tau=tau,
                lifetimes_groups=S_groups, lifetimes=S_units, feasible=feasible,
                ratio=layer_step_ratio(S_groups, T), s_min=s_min)
