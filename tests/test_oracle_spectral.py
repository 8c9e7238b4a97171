"""Pins for the oracle's scores and schedule (Sec. 3.2, Sec. 4.1, App. G).

Each test checks the oracle against something other than itself: hand-derived
singular energies, closed forms the equations imply, the paper's Lemma
lem:sandwich, brute force over tau, and the paper's printed layer-step
arithmetic.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import spectral as sp

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _matrix(case):
    if "rows" in case:
        return np.array(case["rows"], dtype=np.float64)
    if "eye" in case:
        return case["scale"] * np.eye(case["eye"])
    return np.diag(np.array(case["diag"], dtype=np.float64))


@pytest.mark.parametrize("case", _load("scr_hand_cases.json")["cases"], ids=lambda c: c["name"])
def test_scr_hand_cases(case):
    """SCR from W equals the value implied by hand-derived energies (Eq. scr-reg)."""
    W = _matrix(case)
    eta = 1e-6
    s2 = sp.singular_energies(W)
    assert s2.size == case["d"]
    assert sp.top_k(case["d"]) == case["k"]
    assert float(np.sum(s2[:case["k"]])) == pytest.approx(case["lead"], rel=1e-12, abs=1e-9)
    assert sp.frobenius_sq(W) == pytest.approx(case["fro2"], rel=1e-15)
    want = math.log((case["lead"] + eta * case["fro2"]) / (case["tail"] + eta * case["fro2"]))
    assert sp.scr_eta(W, eta) == pytest.approx(want, rel=1e-10, abs=1e-10)


def test_top_k_table():
    g = _load("scr_hand_cases.json")["top_k"]
    assert [sp.top_k(d) for d in g["d"]] == g["k"]


def test_scr_rank_deficient_is_log_one_plus_eta_over_eta():
    """The paper's d = 1 / rank-deficient edge case: with no tail energy the ratio
    is (1 + eta) / eta (Sec. 3.2, remark after Eq. scr-reg)."""
    for eta in (1e-6, 1e-3, 0.5):
        row = np.array([[0.5, -2.0, 7.0]])
        assert sp.scr_eta(row, eta) == pytest.approx(math.log((1 + eta) / eta), rel=1e-12)
        rank1 = np.outer([1.0, -1.0, 2.0, 0.5], [3.0, 1.0, -2.0, 0.25, 4.0, 1.0])
        assert sp.scr_eta(rank1, eta) == pytest.approx(math.log((1 + eta) / eta), rel=1e-9)


@pytest.mark.parametrize("shape,alpha", [((40, 40), 0.3), ((64, 24), 1.0), ((17, 90), 1.5),
                                         ((130, 60), 0.7)])
def test_scr_on_constructed_spectrum(shape, alpha):
    """W = U diag(s) V^T with known s: the oracle recovers the spectrum (float64, 1e-10)."""
    rng = np.random.default_rng(7)
    m, n = shape
    d = min(m, n)
    s = np.arange(1, d + 1, dtype=np.float64) ** (-alpha) * 3.0
    U, _ = np.linalg.qr(rng.standard_normal((m, d)))
    V, _ = np.linalg.qr(rng.standard_normal((n, d)))
    W = (U * s) @ V.T
    eta = 1e-6
    k = sp.top_k(d)
    f2 = float(np.sum(s ** 2))
    want = math.log((np.sum(s[:k] ** 2) + eta * f2) / (np.sum(s[k:] ** 2) + eta * f2))
    assert sp.scr_eta(W, eta) == pytest.approx(want, rel=1e-10)
    np.testing.assert_allclose(sp.singular_energies(W), s ** 2, rtol=1e-9, atol=1e-12)


def test_matrix_score_identity_g_squared():
    """g(W)^2 = (E_k + eta F) / (1 + 2 eta): rho(SCR) = num / (num + den) with
    num + den = F (1 + 2 eta), so F rho = (E_k + eta F) / (1 + 2 eta)."""
    rng = np.random.default_rng(3)
    for eta in (1e-6, 0.1):
        for shape in ((30, 50), (50, 30), (12, 12)):
            W = rng.standard_normal(shape) * rng.uniform(0.1, 3)
            s2 = np.linalg.svd(W, compute_uv=False) ** 2
            k = sp.top_k(min(shape))
            F = np.sum(W * W)
            want = (np.sum(s2[:k]) + eta * F) / (1 + 2 * eta)
            assert sp.matrix_score(W, eta) ** 2 == pytest.approx(want, rel=1e-10)


def test_lemma_sandwich_random():
    """Lemma lem:sandwich with the unregularised ratio: ||W||_F sqrt(rho/k) <= ||W||_2
    <= ||W||_F sqrt(rho), rho = E_k / ||W||_F^2; ||W||_2 from LAPACK's SVD."""
    rng = np.random.default_rng(11)
    for trial in range(300):
        m, n = rng.integers(1, 40, size=2)
        W = rng.standard_normal((m, n)) * (np.arange(1, n + 1) ** -rng.uniform(0, 2))
        s2 = sp.singular_energies(W)
        k = sp.top_k(s2.size)
        F = sp.frobenius_sq(W)
        ek = float(np.sum(s2[:k]))
        if not (0 < ek < F * (1 - 1e-12)):
            continue
        # rho(u) with u = log(E_k / (F - E_k)) through the oracle's logistic
        rho = sp.logistic(math.log(ek / (F - ek)))
        spec = np.linalg.norm(W, 2)
        assert math.sqrt(F) * math.sqrt(rho / k) <= spec * (1 + 1e-9)
        assert spec <= math.sqrt(F) * math.sqrt(rho) * (1 + 1e-9)


def test_logistic_values():
    assert sp.logistic(0.0) == 0.5
    assert sp.logistic(math.log(3.0)) == pytest.approx(0.75, rel=1e-15)
    assert sp.logistic(-math.log(3.0)) == pytest.approx(0.25, rel=1e-15)
    assert sp.logistic(800.0) == 1.0 and sp.logistic(-800.0) == 0.0


def _r(eta):
    # g(x I_10) / x = sqrt((1 + 10 eta) / (1 + 2 eta)), derived by hand: sigma^2 = x^2 (10
    # times), k = 1, rho = (1 + 10 eta) / (10 (1 + 2 eta)), F = 10 x^2.
    return math.sqrt((1 + 10 * eta) / (1 + 2 * eta))


def test_attention_score_roles():
    """Eq. app-attn-score on scaled identities: Q=1, K=2, V=3, O=4 (x I_10), d_h = 4.
    Swapping the value/output pair with the query/key pair changes the result."""
    eta = 1e-6
    I = np.eye(10)
    r = _r(eta)
    got = sp.attn_score(1 * I, 2 * I, 3 * I, 4 * I, d_head=4, eta=eta)
    want = (4 * r) * (3 * r) * (1 + (1 * r) * (2 * r) / 2.0)
    assert got == pytest.approx(want, rel=1e-12)
    swapped = sp.attn_score(3 * I, 4 * I, 1 * I, 2 * I, d_head=4, eta=eta)
    assert abs(swapped - got) > 1.0


def test_mlp_score_hand():
    """Eq. app-mlp-score: W_1 = p [I; I] (20 x 10), W_2 = w I_10.
    g(W_1) = p sqrt(2) r and g(W_2) = w r by the same hand derivation."""
    eta = 1e-6
    r = _r(eta)
    p, w = 1.5, 0.25
    W1 = p * np.vstack([np.eye(10), np.eye(10)])
    W2 = w * np.eye(10)
    assert sp.mlp_score(W1, W2, eta) == pytest.approx(p * math.sqrt(2) * r * w * r, rel=1e-12)


def test_unit_scores_sum_and_normalise():
    """Eq. app-block-score sums the submodule scores; Eq. app-score-normalization
    divides by max + 1e-12."""
    bq = [1.0, 2.0, 5.0, 0.5, 3.0, 3.0]
    q = sp.unit_scores(bq, [0, 0, 1, 1, 2, 2])
    np.testing.assert_array_equal(q, [3.0, 5.5, 6.0])
    lam = sp.normalise(q)
    assert lam[2] == 6.0 / (6.0 + 1e-12)
    assert lam[2] < 1.0 and 1.0 - lam[2] < 1e-12
    assert lam[0] == pytest.approx(0.5, rel=1e-12)


def test_lifetime_rule_cases():
    """Eq. schedule: S = max(S_min, ceil(T min(1, lam / tau)))."""
    lam = np.array([1.0, 0.5, 0.26, 0.01, 0.0])
    S = sp.lifetimes(lam, T=10, tau=1.0, s_min=1)
    np.testing.assert_array_equal(S, [10, 5, 3, 1, 1])
    S = sp.lifetimes(lam, T=10, tau=0.5, s_min=2)
    np.testing.assert_array_equal(S, [10, 10, 6, 2, 2])
    S = sp.lifetimes(lam, T=100, tau=2.0, s_min=10)
    np.testing.assert_array_equal(S, [50, 25, 13, 10, 10])


def test_min_lifetime_reading():
    assert [sp.min_lifetime(T) for T in (4, 10, 30, 50, 64, 100)] == [1, 1, 3, 5, 6, 10]


def _brute_best(lam, T, budget, s_min):
    """Dense log grid of tau plus points just around every breakpoint."""
    cap = sp.budget_cap(budget, len(lam), T)
    taus = list(np.geomspace(1e-4, 1e4, 20000))
    for x in lam:
        for j in range(1, T + 1):
            b = T * x / j
            taus += [b * (1 - 1e-9), b * (1 + 1e-9)]
    best = None
    for tau in taus:
        S = sp.lifetimes(lam, T, tau, s_min)
        if S.sum() <= cap and (best is None or S.sum() > best.sum()):
            best = S
    return best


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("budget", [1.0, 0.5, 0.33])
def test_budget_rule_matches_brute_force(seed, budget):
    rng = np.random.default_rng(seed)
    G, T = int(rng.integers(2, 7)), int(rng.choice([4, 10, 16]))
    lam = sp.normalise(rng.uniform(0.05, 1.0, size=G))
    s_min = sp.min_lifetime(T)
    tau, S, ok = sp.tau_for_budget(lam, T, budget, s_min)
    assert ok
    want = _brute_best(lam, T, budget, s_min)
    np.testing.assert_array_equal(S, want)
    np.testing.assert_array_equal(sp.lifetimes(lam, T, tau, s_min), S)


def test_budget_full_is_all_T_and_monotone_in_score():
    """100% budget gives S_l = T for every unit; Corollary cor:safe: a lower score
    never gets a longer lifetime."""
    rng = np.random.default_rng(5)
    lam = sp.normalise(rng.uniform(0.01, 1.0, size=32))
    for T in (10, 64):
        _, S, _ = sp.tau_for_budget(lam, T, 1.0, sp.min_lifetime(T))
        assert np.all(S == T)
        for budget in (0.5, 0.33):
            _, S, _ = sp.tau_for_budget(lam, T, budget, sp.min_lifetime(T))
            order = np.argsort(lam)
            assert np.all(np.diff(S[order]) >= 0)
            assert S.sum() <= sp.budget_cap(budget, 32, T)


def test_budget_infeasible_falls_back_to_s_min():
    lam = np.array([1.0, 0.9, 0.8])
    tau, S, ok = sp.tau_for_budget(lam, 10, 0.05, 1)
    assert not ok and math.isinf(tau) and np.all(S == 1)


def test_paper_layer_step_arithmetic():
    """Table tab:kernel: 3200 layer-steps for 32 layers x T=100, 1120 scheduled = 35%;
    the budget rule at 35% on 32 layers x T=100 spends at most 1120 layer-steps."""
    g = _load("paper_arithmetic.json")
    assert g["layers"] * g["T"] == g["full_layer_steps"]
    assert Fraction(g["scheduled_layer_steps"], g["full_layer_steps"]) == Fraction(35, 100)
    assert round(1 / g["budget"], 2) == g["ceiling_speedup"]
    rng = np.random.default_rng(0)
    lam = sp.normalise(rng.uniform(0.05, 1.0, size=g["layers"]))
    _, S, ok = sp.tau_for_budget(lam, g["T"], g["budget"], sp.min_lifetime(g["T"]))
    assert ok
    assert S.sum() <= g["scheduled_layer_steps"]
    assert S.sum() >= g["scheduled_layer_steps"] - g["layers"]  # within one step per layer
    assert sp.layer_step_ratio(S, g["T"]) <= g["budget"]


def test_active_sets_nested_and_group_closed():
    S_groups = np.array([3, 1, 4, 4])
    groups = [0, 0, 1, 1, 2, 2, 3, 3]
    S_units = [S_groups[g] for g in groups]
    A = sp.active_sets(S_units, T=4)
    # A_1 is everything; sets only shrink
    assert A[0].all()
    assert np.all(A[1:] <= A[:-1])
    # members of a group are active together
    for g in range(4):
        members = [u for u, gg in enumerate(groups) if gg == g]
        assert np.all(A[:, members] == A[:, members[:1]])
    # row sums equal the number of units with S >= s
    for s in range(1, 5):
        assert A[s - 1].sum() == sum(1 for x in S_units if x >= s)


# ---------------------------------------------------------------------------
# alternative static rankings (Table tab:cross-ablation)
# ---------------------------------------------------------------------------

def test_matrix_statistics_on_known_spectra():
    """diag(s) and U diag(s) V^T with known s: ||W||_F^2 = sum s^2, ||W||_2 = max s, stable
    rank = sum s^2 / max s^2, the product, raw SCR = Eq. scr-reg from s."""
    rng = np.random.default_rng(11)
    s = np.array([5.0, 3.0, 2.0, 1.0, 0.5, 0.25, 0.1, 0.1, 0.05, 0.01, 0.01, 0.003])
    U, _ = np.linalg.qr(rng.standard_normal((20, 12)))
    V, _ = np.linalg.qr(rng.standard_normal((12, 12)))
    for W in (np.diag(s), (U * s) @ V.T, ((U * s) @ V.T).T):
        f2 = float(np.sum(s ** 2))
        assert sp.matrix_statistic(W, "frobenius") == pytest.approx(math.sqrt(f2), rel=1e-12)
        assert sp.matrix_statistic(W, "spectral") == pytest.approx(5.0, rel=1e-10)
        assert sp.matrix_statistic(W, "stable_rank") == pytest.approx(f2 / 25.0, rel=1e-10)
        assert sp.matrix_statistic(W, "frob_stable_rank") == pytest.approx(math.sqrt(f2) * f2 / 25.0,
                                                                          rel=1e-10)
        eta = 1e-6
        want = math.log((25.0 + eta * f2) / (f2 - 25.0 + eta * f2))  # k = 1 for d = 12
        assert sp.matrix_statistic(W, "raw_scr") == pytest.approx(want, rel=1e-10)
        assert sp.matrix_statistic(W, "scr") == sp.matrix_score(W)


def _scaled_identity_model():
    """Two-block pre-norm model whose projections are diagonal with known entries, so that
    every statistic has a closed form: W_Q, W_K, W_V, W_O = diag(a_j), j = 1..4, per block;
    W_1 = [diag(p); diag(p)] (gated), W_2 = diag(w)."""
    from paper_2609_29505_gb300 import synth
    cfg = synth.ModelConfig(name="ranks", stem="time_add", block="prenorm", norm="rms",
                            mlp="swiglu", head="linear", n_blocks=2, d=4, n_heads=1, d_head=4,
                            d_ff=4, batch=1, n_tokens=2, d_in=4, d_out=4, out_channels=4, T=4)
    base = np.array([1.0, 0.5, 0.25, 0.125])
    W = {}
    for b in range(2):
        a = [(b + 1) * j * base for j in (1, 2, 3, 4)]
        W[f"blocks.{b}.w_qkv"] = np.vstack([np.diag(a[0]), np.diag(a[1]), np.diag(a[2])])
        W[f"blocks.{b}.w_o"] = np.diag(a[3])
        W[f"blocks.{b}.w_1"] = np.vstack([np.diag(1.5 * base), np.diag(1.5 * base)])
        W[f"blocks.{b}.w_2"] = np.diag((b + 2) * base)
    return cfg, W, base


@pytest.mark.parametrize("ranking", ["frobenius", "spectral", "stable_rank", "frob_stable_rank"])
def test_ranked_branch_scores_hand_model(ranking):
    """Branch formulas of App. G with the ranking's statistic, derived by hand: for
    c diag(base), ||.||_F = c n2, ||.||_2 = c, stable rank = n2^2 (n2 = ||base||); the
    stacked [diag(p); diag(p)] doubles the squared Frobenius norm."""
    cfg, W, base = _scaled_identity_model()
    n2 = math.sqrt(float(np.sum(base ** 2)))
    stat = {"frobenius": lambda c, k=1: c * n2 * math.sqrt(k),
            "spectral": lambda c, k=1: c * math.sqrt(k),
            "stable_rank": lambda c, k=1: n2 ** 2,
            "frob_stable_rank": lambda c, k=1: c * n2 * math.sqrt(k) * n2 ** 2}[ranking]
    want = []
    for b in range(2):
        gq, gk, gv, go = (stat((b + 1) * j) for j in (1, 2, 3, 4))
        want.append(go * gv * (1.0 + gq * gk / 2.0))
        want.append(stat(b + 2) * stat(1.5, 2))
    got = sp.ranked_branch_scores(cfg, W, ranking)
    np.testing.assert_allclose(got, want, rtol=1e-10)


def test_ranked_branch_scores_depth_random_and_scr():
    cfg, W, _ = _scaled_identity_model()
    assert sp.ranked_branch_scores(cfg, W, "depth") == [4.0, 3.0, 2.0, 1.0]
    draws = [0.3, 0.9, 0.1, 0.5]
    assert sp.ranked_branch_scores(cfg, W, "random", draws=draws) == draws
    with pytest.raises(ValueError):
        sp.ranked_branch_scores(cfg, W, "random")
    np.testing.assert_allclose(sp.ranked_branch_scores(cfg, W, "scr"), sp.branch_scores(cfg, W),
                               rtol=1e-15)
