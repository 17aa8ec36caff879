"""Pins for the oracle's cutoff design (Section 3.3, Appendices D and F, Section 4 variants)."""
import math

import numpy as np
import pytest
from scipy.optimize import minimize

from oracle import design
from oracle.cutoffs import ONE62, cumulative_masses, inverse_survival_weights, sample_cutoffs


def _objective(w, xi):
    return float(np.sum(np.asarray(w) / np.asarray(xi)))


def _brute(w, B, cap):
    """The design problem solved by a general constrained solver (SLSQP). Monotonicity holds by
    construction: xi_t = sum_{j >= t} y_j with y >= 0."""
    T = len(w)
    to_xi = lambda y: np.cumsum(y[::-1])[::-1]  # noqa: E731
    cons = [{"type": "eq", "fun": lambda y: np.sum(to_xi(y)) - B}]
    if cap:
        cons.append({"type": "ineq", "fun": lambda y: 1.0 - np.sum(y)})
    best = None
    for start_xi in (np.full(T, B / T), np.linspace(1.6, 0.4, T) * B / T, np.linspace(1.2, 0.8, T) * B / T):
        if cap:
            start_xi = np.minimum(start_xi, 1.0)
        y0 = np.maximum(np.append(-np.diff(start_xi), start_xi[-1]), 1e-6)
        for method, opts in (("SLSQP", {"ftol": 1e-15, "maxiter": 5000}),
                             ("trust-constr", {"xtol": 1e-14, "gtol": 1e-12, "maxiter": 20000})):
            r = minimize(lambda y: _objective(w, to_xi(y)), y0, method=method, bounds=[(1e-12, None)] * T,
                         constraints=cons, options=opts)
            feasible = abs(np.sum(to_xi(r.x)) - B) < 1e-9 and np.all(r.x >= -1e-12) and \
                (not cap or np.sum(r.x) <= 1.0 + 1e-9)
            if feasible and (best is None or r.fun < best.fun):    # SLSQP's success flag is often
                best = r                                            # spuriously false at the optimum
    assert best is not None
    best.x = to_xi(best.x)
    return best


@pytest.mark.filterwarnings("ignore:delta_grad == 0.0")      # the reference solver's quasi-Newton notice
@pytest.mark.parametrize("seed", range(8))
def test_pav_matches_a_general_solver(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(3, 8))
    w = rng.uniform(0.05, 3.0, T) ** 2
    B = float(rng.uniform(0.3, 0.9) * T) if seed % 2 else float(rng.uniform(0.1, 0.4) * T)
    xi = design.monotone_design(w, B)
    assert np.all(np.diff(xi) <= 1e-15) and abs(xi.sum() - B) < 1e-12
    ref = _brute(w, B, cap=False)
    assert _objective(w, xi) <= ref.fun * (1 + 1e-7)
    np.testing.assert_allclose(xi, ref.x, rtol=2e-4, atol=2e-5)


@pytest.mark.filterwarnings("ignore:delta_grad == 0.0")
@pytest.mark.parametrize("seed", range(6))
def test_capped_design_matches_a_general_solver(seed):
    rng = np.random.default_rng(100 + seed)
    T = int(rng.integers(3, 8))
    w = np.sort(rng.uniform(0.1, 4.0, T))[::-1] ** 3          # steep front weights force saturation
    w[rng.integers(0, T)] *= 5.0                               # plus a violation to pool
    B = float(rng.uniform(0.6, 0.95) * T)
    xi = design.capped_monotone_design(w, B)
    assert np.all(xi <= 1.0 + 1e-15) and np.all(np.diff(xi) <= 1e-15) and abs(xi.sum() - B) < 1e-12
    ref = _brute(w, B, cap=True)
    assert _objective(w, xi) <= ref.fun * (1 + 1e-7)
    np.testing.assert_allclose(xi, ref.x, rtol=2e-4, atol=2e-5)


def test_closed_form_special_cases():
    # already non-increasing sqrt(w): no pooling, the unconstrained closed form is the answer
    w = np.array([9.0, 4.0, 4.0, 1.0])
    np.testing.assert_allclose(design.monotone_design(w, 2.0), 2.0 * np.sqrt(w) / np.sqrt(w).sum(), rtol=1e-15)
    np.testing.assert_allclose(design.closed_form(w, 2.0), [2 * 3 / 8, 2 * 2 / 8, 2 * 2 / 8, 2 * 1 / 8])
    # increasing weights pool into one block: uniform xi = B / T
    np.testing.assert_allclose(design.monotone_design(np.array([1.0, 2.0, 3.0, 4.0]), 2.0), 0.5, rtol=1e-15)
    # a single violating pair pools to sqrt of its mean weight
    xi = design.monotone_design(np.array([4.0, 1.0, 9.0]), 1.0)
    s = [2.0, math.sqrt(5.0), math.sqrt(5.0)]     # blocks [4] | [1, 9] -> 2 < sqrt(5): all pool
    assert xi[0] == pytest.approx(xi[1]) == pytest.approx(xi[2])
    assert s[0] < s[1]


def test_time_prior_and_uniform_and_fixed():
    xi = design.time_prior_design(500, 64.0)
    assert abs(xi.sum() - 64.0) < 1e-9 and xi[0] == 1.0 and np.all(np.diff(xi) < 0)
    lam = -math.log(xi[1])
    np.testing.assert_allclose(xi, np.exp(-lam * np.arange(500)), rtol=1e-12)
    u = design.uniform_design(10)
    assert u[0] == 1.0 and u[-1] == pytest.approx(0.1) and u.sum() == pytest.approx(5.5)   # E[H] = (T+1)/2
    f = design.fixed_prefix_design(10, 4)
    assert list(f) == [1, 1, 1, 1, 0, 0, 0, 0, 0, 0]
    h = design.heuristic_design(np.array([1.0, 4.0, 0.25, 1.0]), 2.0)
    assert np.all(np.diff(h) <= 0) and np.all(h <= 1.0)


def test_masses_realise_xi_and_the_budget():
    rng = np.random.default_rng(3)
    w = rng.uniform(0.1, 2.0, 300) ** 2
    xi = design.capped_monotone_design(w, 40.0)
    q = design.masses_from_xi(xi)
    U = cumulative_masses(q)
    assert U[-1] <= ONE62
    # Pr(H = 0) = 1 - xi_1; Pr(H >= t) = xi_t up to the 2^-62 quantisation; E[H] = sum xi = B
    assert abs((ONE62 - U[-1]) / ONE62 - (1.0 - xi[0])) < 1e-15 * 300
    real = np.array([(U[-1] - U[t - 1]) / ONE62 for t in range(1, 301)])
    np.testing.assert_allclose(real, xi, rtol=1e-12, atol=1e-15 * 300)
    EH = sum((h + 1) * int(m) for h, m in enumerate(q)) / ONE62
    assert EH == pytest.approx(40.0, rel=1e-12)


def test_zero_cutoff_mode_draws_h0_with_the_deficit():
    T, M = 12, 4000
    xi = design.monotone_design(np.ones(T), 3.0)          # uniform xi = 0.25
    q = design.masses_from_xi(xi)[None]
    L = np.full(1, T, dtype=np.int32)
    Hs = np.array([sample_cutoffs(q, L, 1, seed=1, step=s, mode="trunc_zero")[0][0] for s in range(M)])
    p0 = (Hs == 0).mean()
    assert abs(p0 - 0.75) < 4.5 * math.sqrt(0.75 * 0.25 / M)
    w = inverse_survival_weights(q[0], allow_zero=True)
    np.testing.assert_allclose(w, 4.0, rtol=1e-12)
    with pytest.raises(ValueError):
        sample_cutoffs(q, L, 1, seed=1, step=0, mode="trunc")    # the exact mode insists on 2^62


def test_group_mean_by_step_by_hand():
    L = np.array([3, 1, 2, 2])
    vals = np.array([1., 2., 3., 10., 5., 6., 7., 8.])
    g = design.group_mean_by_step(vals, L, 2)
    np.testing.assert_allclose(g, [[(1 + 10) / 2, 2 / 2, 3 / 2], [(5 + 7) / 2, (6 + 8) / 2, 0.0]])


def test_score_proxy_is_the_squared_head_gradient_norm():
    # gamma = || d log p(o) / dW ||_F^2, checked by central differences over every entry of W
    rng = np.random.default_rng(7)
    d, V = 3, 5
    H = rng.standard_normal((4, d))
    W = rng.standard_normal((V, d)) * 0.7
    tok = np.array([0, 4, 2, 2])
    gamma, logp = design.score_proxy(H, W, tok)
    eps = 1e-6
    for i in range(4):
        def lp(Wm):
            z = Wm @ H[i]
            return z[tok[i]] - (z.max() + math.log(np.exp(z - z.max()).sum()))
        g = np.zeros_like(W)
        for v in range(V):
            for c in range(d):
                Wp, Wn = W.copy(), W.copy()
                Wp[v, c] += eps
                Wn[v, c] -= eps
                g[v, c] = (lp(Wp) - lp(Wn)) / (2 * eps)
        assert gamma[i] == pytest.approx(float((g * g).sum()), rel=1e-7)
        assert logp[i] == pytest.approx(lp(W), rel=1e-13)


def _u_full(L, K, R, P_rows):
    """Eq. ut_def with the full next-token distributions (no top-k)."""
    V = P_rows.shape[1]
    idx = np.tile(np.arange(V), (P_rows.shape[0], 1))
    return design.reward_uncertainty(L, K, R, idx, P_rows)


def test_uncertainty_closed_cases():
    L = np.array([3, 3, 3, 3])
    V = 4
    one = np.zeros((12, V))
    one[:, 1] = 1.0
    # every completion succeeds: the reward is certain, u = 0
    assert np.all(_u_full(L, 4, np.ones(4), one) == 0.0)
    # half succeed but all predict the same distribution: nothing separates them, u = 1/2
    assert np.allclose(_u_full(L, 4, np.array([1, 1, 0, 0]), one), 0.5)
    # successes put their mass on token 0, failures on token 3: the prefix decides the reward, u = 0
    sep = np.zeros((12, V))
    sep[0:6, 0] = 1.0
    sep[6:12, 3] = 1.0
    assert np.allclose(_u_full(L, 4, np.array([1, 1, 0, 0]), sep), 0.0)
    # Bernoulli bound: u <= 1/2 always, and min(p_hat, 1 - p_hat) <= ... >= 0
    rng = np.random.default_rng(0)
    Pr = rng.dirichlet(np.ones(V), size=12)
    u = _u_full(L, 4, np.array([1, 0, 0, 0]), Pr)
    assert np.all((u >= 0) & (u <= 0.5))


def test_topk_route_with_every_token_is_the_definition():
    rng = np.random.default_rng(5)
    K, V = 4, 12
    L = rng.integers(2, 7, size=2 * K)
    R = np.array([1, 0, 1, 1, 0, 0, 1, 0], dtype=np.float32)
    H = rng.standard_normal((int(L.sum()), 3))
    W = rng.standard_normal((V, 3)) * 1.3
    idx_full, p_full = design.topk_policy(H, W, V)
    u_full = design.reward_uncertainty(L, K, R, idx_full, p_full)
    # with k = V the top-k route equals the definition written with full distributions
    z = H @ W.T
    Pr = np.exp(z - z.max(axis=1, keepdims=True))
    Pr /= Pr.sum(axis=1, keepdims=True)
    np.testing.assert_allclose(u_full, _u_full(L, K, R, Pr), atol=1e-14)
    # dropping only tokens of zero probability changes nothing
    Pr2 = np.concatenate([Pr, np.zeros((Pr.shape[0], 5))], axis=1)
    np.testing.assert_allclose(_u_full(L, K, R, Pr2), u_full, atol=1e-14)
    # and u stays within [0, 1/2] for every k
    for k in (1, 3, 6):
        idx, pk = design.topk_policy(H, W, k)
        uk = design.reward_uncertainty(L, K, R, idx, pk)
        assert np.all((uk >= 0) & (uk <= 0.5))


def test_topk_policy_orders_and_ties():
    W = np.array([[1.0], [3.0], [3.0], [0.5]])
    idx, p = design.topk_policy(np.array([[1.0]]), W, 3)
    assert list(idx[0]) == [1, 2, 0]
    assert p[0, 0] == pytest.approx(p[0, 1]) and p[0].sum() < 1.0


def test_sigmoid_recipe_is_the_logistic_function():
    # Appendix G's sigma(r) = 1 / (1 + e^-r): against the library exponential, its symmetry and
    # its fixed points
    r = np.linspace(-40.0, 40.0, 40001)
    got = np.array([design.sigmoid_recipe(x) for x in r])
    ref = 1.0 / (1.0 + np.exp(-r))
    assert np.max(np.abs(got - ref) / ref) < 1e-14
    assert np.max(np.abs(got + got[::-1] - 1.0)) < 4e-15          # sigma(-r) = 1 - sigma(r)
    assert np.all(np.diff(got) >= 0.0)
    assert design.sigmoid_recipe(0.0) == 0.5
    assert design.sigmoid_recipe(float("inf")) == design.sigmoid_recipe(1e9) == design.sigmoid_recipe(40.0)
    assert design.sigmoid_recipe(float("nan")) == 0.0


@pytest.mark.parametrize("r", [-3.0, -0.5, 0.0, 0.8, 2.5])
def test_binarized_labels_are_bernoulli_sigma(r):
    # y ~ Bernoulli(sigma(r)): the label frequency over many trajectories is sigma(r)
    M = 4000
    y = design.binarize_rewards(np.full(M, r, dtype=np.float32), seed=11, step=2)
    assert set(np.unique(y)) <= {0.0, 1.0}
    p = 1.0 / (1.0 + math.exp(-r))
    assert abs(y.mean() - p) < 4.5 * math.sqrt(p * (1 - p) / M)


def test_binarized_labels_extremes_and_streams():
    y = design.binarize_rewards(np.array([60.0, -60.0, np.inf, -np.inf, np.nan], dtype=np.float32), 1, 0)
    assert list(y[:1]) == [1.0] and y[2] == 1.0 and y[4] == 0.0
    assert y[1] == 0.0 and y[3] == 0.0        # a label 1 would need the uniform to be exactly 0
    # a shard starting at trajectory 7 draws what the whole batch draws for its trajectories
    R = np.random.default_rng(0).normal(0, 2, 20).astype(np.float32)
    whole = design.binarize_rewards(R, 5, 3)
    assert np.array_equal(design.binarize_rewards(R[7:], 5, 3, traj_base=7), whole[7:])
    assert not np.array_equal(design.binarize_rewards(R, 5, 4), whole)    # the step changes the draw


def test_non_finite_weights_are_refused():
    with pytest.raises(ValueError):
        design.timestep_weights(np.array([1.0, np.nan, 2.0]), None)
    with pytest.raises(ValueError):
        design.timestep_weights(np.array([1.0, 2.0]), np.array([np.inf, 0.1]))


# ---------------------------------------------------------------- the whole design step, by hand
def _two_prompt_batch():
    """Prompt 0: lengths (4, 2), per-token scores (16, 4, 8, 2) and (16, 4), so gamma_bar =
    (16, 4, 4, 1) over T_0 = 4 (the short completion adds 0 beyond its end) and sqrt(w) =
    (4, 2, 2, 1), sum 9. Prompt 1: lengths (2, 1), T_1 = 2 < T_max = 4."""
    L = np.array([4, 2, 2, 1], dtype=np.int32)
    gamma_full = np.array([16., 4., 8., 2.,  16., 4.,  5., 3.,  7.])
    return L, gamma_full


def test_design_masses_per_prompt_horizon_and_budget_by_hand():
    L, g = _two_prompt_batch()
    # budget 2: prompt 0 takes the closed form 2 (4, 2, 2, 1) / 9 (already non-increasing, below
    # the cap); prompt 1's budget is min(2, T_1) = 2 = T_1, so xi = (1, 1) and H = L surely
    q, xi = design.design_cutoff_masses(L, 2, g, None, 2.0, "optimized")
    np.testing.assert_allclose(xi[0], [8 / 9, 4 / 9, 4 / 9, 2 / 9], rtol=1e-15)
    assert list(xi[1]) == [1.0, 1.0, 0.0, 0.0]
    # masses: Pr(H = h) = xi_h - xi_{h+1}; Pr(H = 0) = 1 - xi_1 = 1/9 is the deficit
    np.testing.assert_allclose(q[0].astype(np.float64) / ONE62, [4 / 9, 0.0, 2 / 9, 2 / 9], rtol=1e-15, atol=0)
    assert int(q[0, 1]) == 0
    assert abs((ONE62 - sum(int(x) for x in q[0])) / ONE62 - 1 / 9) < 1e-15
    assert [int(x) for x in q[1]] == [0, ONE62, 0, 0]          # zero beyond T_1, no deficit


def test_design_masses_cap_and_budget_above_the_horizon():
    L, g = _two_prompt_batch()
    # budget 3.5: prompt 0's closed form starts at 3.5 * 4 / 9 > 1, so the cap saturates xi_1 and
    # the suffix (w = 4, 4, 1; sqrt 2, 2, 1, sum 5) gets budget 2.5: (1, 1, 0.5). Prompt 1: the
    # budget exceeds T_1 = 2 and becomes 2 (a budget above the horizon has no design).
    q, xi = design.design_cutoff_masses(L, 2, g, None, 3.5, "optimized")
    np.testing.assert_allclose(xi[0], [1.0, 1.0, 1.0, 0.5], rtol=1e-15)
    assert list(xi[1]) == [1.0, 1.0, 0.0, 0.0]
    assert [int(x) for x in q[0]] == [0, 0, ONE62 // 2, ONE62 // 2]
    assert [int(x) for x in q[1]] == [0, ONE62, 0, 0]
    with pytest.raises(ValueError):
        design.capped_monotone_design([1.0, 1.0], 3.5)           # what B in place of min(B, T_p) would do


def test_design_masses_use_u_per_prompt():
    L, g = _two_prompt_batch()
    # u scales the weights step by step: gamma_bar_0 = (16, 4, 4, 1) times u_0 = (1/4, 1, 1/4, 1)
    # gives w = (4, 4, 1, 1), sqrt (2, 2, 1, 1), sum 6; budget 2: (2/3, 2/3, 1/3, 1/3)
    u = np.array([[0.25, 1.0, 0.25, 1.0], [1.0, 1.0, 0.0, 0.0]])
    _, xi = design.design_cutoff_masses(L, 2, g, u, 2.0, "optimized")
    np.testing.assert_allclose(xi[0], [2 / 3, 2 / 3, 1 / 3, 1 / 3], rtol=1e-15)


def test_design_masses_other_strategies_by_hand():
    L, g = _two_prompt_batch()
    q, xi = design.design_cutoff_masses(L, 2, g, None, 2.0, "uniform")
    np.testing.assert_allclose(xi[0], [1.0, 0.75, 0.5, 0.25], rtol=1e-15)
    assert [int(x) for x in q[0]] == [ONE62 // 4] * 4
    assert [int(x) for x in q[1]] == [ONE62 // 2, ONE62 // 2, 0, 0]
    q, xi = design.design_cutoff_masses(L, 2, g, None, 2.0, "fixed", param=2)
    assert list(xi[0]) == [1.0, 1.0, 0.0, 0.0] and [int(x) for x in q[0]] == [0, ONE62, 0, 0]
    assert list(xi[1]) == [1.0, 1.0, 0.0, 0.0]
    q, xi = design.design_cutoff_masses(L, 2, g, None, 2.0, "heuristic")
    np.testing.assert_allclose(xi[0], [8 / 9, 4 / 9, 4 / 9, 2 / 9], rtol=1e-15)
    q, xi = design.design_cutoff_masses(L, 2, g, None, 2.0, "time_prior")
    assert list(xi[1]) == [1.0, 1.0, 0.0, 0.0]                  # budget = T_1: lambda = 0
    assert abs(xi[0].sum() - 2.0) < 1e-12 and xi[0][0] == 1.0


def test_timestep_weight_floor_and_all_zero_rule():
    w = design.timestep_weights(np.array([4.0, 0.0, 1.0]), None)
    assert w == [4.0, 4.0 * design.W_FLOOR, 1.0]
    w = design.timestep_weights(np.array([2.0, 3.0]), np.array([0.5, 0.0]))
    assert w == [1.0, design.W_FLOOR]
    assert design.timestep_weights(np.zeros(3), None) == [1.0, 1.0, 1.0]
    assert design.timestep_weights(np.array([1.0, 2.0]), np.zeros(2)) == [1.0, 1.0]
    # a weight already above the floor is kept as it is
    assert design.timestep_weights(np.array([1.0, 2e-12]), None) == [1.0, 2e-12]


def test_heuristic_cap_and_running_minimum_by_hand():
    # closed form 3.5 (4, 2, 2, 1) / 9 starts above 1: the cap clips xi_1 only (the heuristic does
    # not hand the clipped mass back, so its total falls below the budget)
    h = design.heuristic_design(np.array([16.0, 4.0, 4.0, 1.0]), 3.5)
    np.testing.assert_allclose(h, [1.0, 7 / 9, 7 / 9, 3.5 / 9], rtol=1e-15)
    # sqrt(w) = (1, 4, 2): closed form (1, 4, 2) / 7, then the running minimum holds 1/7
    h = design.heuristic_design(np.array([1.0, 16.0, 4.0]), 1.0)
    np.testing.assert_allclose(h, [1 / 7, 1 / 7, 1 / 7], rtol=1e-15)
