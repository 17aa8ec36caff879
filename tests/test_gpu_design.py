"""Parity of the cutoff-design step (score proxy, design, H = 0 sampling) with the oracle.

The design kernel and the oracle get the same seeded gamma and u, and their masses are compared
bit for bit (both run the same sequence of rounded float64 operations); the time prior, whose
bisection goes through exp(), is compared to 1e-12. The score proxy is compared with the oracle's
float64 softmax within 1e-4 relative.
"""
import numpy as np
import pytest
import torch

from oracle import design
from oracle.cutoffs import sample_cutoffs
from oracle.pipeline import widen
from synthetic import get_config, make_batch
from synthetic.generate import draw_design_inputs, draw_lengths

pytestmark = pytest.mark.gpu

STRAT = {"optimized": 0, "heuristic": 1, "uniform": 2, "time_prior": 3, "fixed": 4}


def _gpu_design(cfg, L, gamma, u, budget, strategy, param=0.0):
    from paper_2606_29758_gb300 import _binding as B
    P, K, T = cfg.P, cfg.K, int(L.max())
    q = torch.empty(P, T, dtype=torch.int64, device="cuda")
    xi = torch.empty(P, T, dtype=torch.float64, device="cuda")
    ws = torch.empty(B.ps_design_cutoffs_workspace_size(P, K, T), dtype=torch.uint8, device="cuda")
    g = torch.from_numpy(gamma).cuda() if gamma is not None else None
    uu = torch.from_numpy(u).cuda() if u is not None else None
    B.ps_design_cutoffs(P, K, T, torch.from_numpy(L).cuda(), g, uu, budget, STRAT[strategy], param, q, xi, ws)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
    return q.cpu().numpy().view(np.uint64), xi.cpu().numpy()


@pytest.mark.parametrize("name,budget", [("mid", 40.0), ("7b", 128.0), ("long", 512.0), ("tiny_bf16", 250.0)])
@pytest.mark.parametrize("strategy", ["optimized", "heuristic", "uniform", "fixed"])
def test_design_masses_bit_exact(name, budget, strategy):
    cfg = get_config(name)
    L = draw_lengths(cfg)
    gamma, u = draw_design_inputs(cfg, L)
    for uu in (u, None):
        q, xi = _gpu_design(cfg, L, gamma, uu, budget, strategy, param=64.0)
        q_ref, xi_ref = design.design_cutoff_masses(L, cfg.K, gamma, uu, budget, strategy, param=64.0)
        assert np.array_equal(xi, xi_ref), np.abs(xi - xi_ref).max()
        assert np.array_equal(q, q_ref)


@pytest.mark.parametrize("name,budget", [("7b", 2048.0), ("long", 8192.0), ("mid", 150.0), ("tiny_bf16", 200.0)])
def test_capped_design_at_budgets_that_saturate_long_prefixes(name, budget):
    # budgets whose designs saturate hundreds to thousands of leading steps at xi = 1 (the cap of
    # Appendix F): the kernel locates the prefix from one pass of pooling from the right and decides
    # the candidates near the cap exactly; the masses must still equal the oracle's linear scan
    cfg = get_config(name)
    L = draw_lengths(cfg)
    gamma, u = draw_design_inputs(cfg, L)
    q, xi = _gpu_design(cfg, L, gamma, u, budget, "optimized")
    q_ref, xi_ref = design.design_cutoff_masses(L, cfg.K, gamma, u, budget, "optimized")
    assert np.array_equal(xi, xi_ref), np.abs(xi - xi_ref).max()
    assert np.array_equal(q, q_ref)
    assert (xi == 1.0).sum() > 0


def _crafted_design(vectors, budget):
    """One prompt per weight vector, each a group of one completion (K = 1), so gamma_bar, and with
    no u the weights, are the vector itself (floored at 1e-12 of the maximum)."""
    from types import SimpleNamespace
    L = np.array([len(v) for v in vectors], dtype=np.int32)
    gamma = np.concatenate([np.asarray(v, dtype=np.float32) for v in vectors])
    q, xi = _gpu_design(SimpleNamespace(P=len(vectors), K=1), L, gamma, None, budget, "optimized")
    q_ref, xi_ref = design.design_cutoff_masses(L, 1, gamma, None, budget, "optimized")
    assert np.array_equal(xi, xi_ref), np.abs(xi - xi_ref).max()
    assert np.array_equal(q, q_ref)
    return xi


def test_capped_design_crafted_cases():
    # (0, 100, 1 x 10) with B = 3.2: saturating nothing already meets the cap (the pooled block
    # {0, 1} starts at 0.94), while saturating one step does not (1.1): qualifying prefixes are not
    # monotone in their length, so the search must not bisect
    xi = _crafted_design([[0.0, 100.0] + [1.0] * 10], 3.2)
    assert xi[0, 0] < 1.0
    # uniform weights: every suffix design starts at exactly B' / T', i.e. at 1 when B = T (the
    # decision sits on the cap); and below it
    for B in (12.0, 11.5, 3.0):
        _crafted_design([[1.0] * 12, [2.0] * 7, [5.0] * 12], B)
    # steep fronts: geometric weights, a plateau, a ramp up, pooled violators after the cap
    rng = np.random.default_rng(7)
    vecs = [[2.0 ** -t for t in range(60)], [50.0] * 5 + [1.0] * 40, list(np.linspace(1, 30, 50)),
            list(np.sort(rng.uniform(0.1, 9.0, 80))[::-1] ** 3 * rng.uniform(0.5, 1.5, 80))]
    for B in (2.0, 10.0, 25.0, 44.0, 59.0, 60.0):
        _crafted_design(vecs, B)


@pytest.mark.parametrize("seed", range(4))
def test_capped_design_random_steep_weights(seed):
    rng = np.random.default_rng(50 + seed)
    vecs = []
    for _ in range(24):
        T = int(rng.integers(2, 400))
        w = np.sort(rng.lognormal(0.0, 2.0, T))[::-1] * rng.lognormal(0.0, 0.5, T)
        vecs.append(w)
    for B in (1.5, 17.0, 130.0, 399.0):
        _crafted_design(vecs, B)


@pytest.mark.parametrize("name,budget", [("mid", 40.0), ("7b", 128.0)])
def test_time_prior_design(name, budget):
    cfg = get_config(name)
    L = draw_lengths(cfg)
    q, xi = _gpu_design(cfg, L, None, None, budget, "time_prior")
    q_ref, xi_ref = design.design_cutoff_masses(L, cfg.K, None, None, budget, "time_prior")
    np.testing.assert_allclose(xi, xi_ref, rtol=1e-12, atol=1e-300)
    for p in range(cfg.P):
        Tp = int(L[p * cfg.K:(p + 1) * cfg.K].max())
        assert xi[p, :Tp].sum() == pytest.approx(min(budget, Tp), rel=1e-9)


def test_optimized_design_budget_and_monotonicity_at_full_size():
    cfg = get_config("7b")
    L = draw_lengths(cfg)
    gamma, u = draw_design_inputs(cfg, L)
    q, xi = _gpu_design(cfg, L, gamma, u, 128.0, "optimized")
    for p in range(cfg.P):
        Tp = int(L[p * cfg.K:(p + 1) * cfg.K].max())
        x = xi[p, :Tp]
        assert np.all(np.diff(x) <= 0) and x[0] <= 1.0 and x[-1] > 0
        assert x.sum() == pytest.approx(min(128.0, Tp), rel=1e-12)
        EH = sum((h + 1) * int(m) for h, m in enumerate(q[p, :Tp])) / float(1 << 62)
        assert EH == pytest.approx(min(128.0, Tp), rel=1e-9)


def test_zero_cutoff_sampling_bit_exact():
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config("7b")
    L = draw_lengths(cfg)
    gamma, u = draw_design_inputs(cfg, L)
    q_ref, _ = design.design_cutoff_masses(L, cfg.K, gamma, u, 64.0, "optimized")
    T = int(L.max())
    H = torch.empty(cfg.B, dtype=torch.int32, device="cuda")
    n = torch.empty_like(H)
    w = torch.empty(cfg.P, T, device="cuda")
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    hits0 = 0
    for step in range(6):
        B.ps_sample_cutoffs(cfg.P, cfg.K, T, torch.from_numpy(q_ref.view(np.int64)).cuda(), torch.from_numpy(L).cuda(),
                            11, step, 0, B.PS_MODE_TRUNC_ZERO, H, n, w, ws)
        torch.cuda.synchronize()
        assert B.ps_workspace_status(ws)[0] == B.PS_OK
        Hr, nr, wr = sample_cutoffs(q_ref, L, cfg.K, 11, step, mode="trunc_zero")
        assert np.array_equal(H.cpu().numpy(), Hr) and np.array_equal(n.cpu().numpy(), nr)
        fin = np.isfinite(wr)
        assert np.array_equal(w.cpu().numpy()[fin], wr[fin].astype(np.float32))
        hits0 += int((Hr == 0).sum())
    # the exact mode refuses masses that leave room for H = 0
    B.ps_sample_cutoffs(cfg.P, cfg.K, T, torch.from_numpy(q_ref.view(np.int64)).cuda(), torch.from_numpy(L).cuda(),
                        11, 0, 0, B.PS_MODE_TRUNC, H, n, w, ws)
    rc, bits = B.ps_workspace_status(ws)
    assert rc == B.PS_ERR_DEVICE_DATA and bits & B.PS_DEV_BAD_PMF


@pytest.mark.parametrize("name,w_scale", [("mid", 1.0), ("mid", 12.0), ("head7b_small", 1.0)])
def test_score_proxy_matches_oracle(name, w_scale):
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config(name, w_std=0.02 * w_scale)
    b = make_batch(cfg, device="cuda")
    hid, W = widen(cfg, b.hid_full), widen(cfg, b.W)
    tok = b.tok_full.copy()
    if w_scale > 1.0:
        # make the chosen token the most likely one for every third row, so p(o) is not small
        z = hid[::3] @ W.T
        tok[::3] = z.argmax(axis=1)
    N = len(tok)
    gamma = torch.empty(N, device="cuda")
    logp = torch.empty(N, device="cuda")
    ws = torch.empty(B.ps_lmhead_score_proxy_workspace_size(N, cfg.d, cfg.V, B.PS_DTYPE_BF16), dtype=torch.uint8,
                     device="cuda")
    B.ps_lmhead_score_proxy(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, b.dev["hid_full"], b.dev["W"],
                            torch.from_numpy(tok).cuda(), gamma, logp, ws)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
    g_ref, lp_ref = design.score_proxy(hid, W, tok)
    g = gamma.cpu().numpy()
    np.testing.assert_allclose(g, g_ref, rtol=2e-4)
    np.testing.assert_allclose(logp.cpu().numpy(), lp_ref, rtol=1e-4, atol=2e-4)
    # the probability part 1 - 2 p(o) + ||p||^2 on its own, where it is far from 1
    hn = (hid ** 2).sum(axis=1)
    part_ref = g_ref / hn
    sel = part_ref < 0.9
    if w_scale > 1.0:
        assert sel.sum() > 10
        np.testing.assert_allclose(g[sel] / hn[sel], part_ref[sel], rtol=2e-4, atol=2e-5)


@pytest.mark.parametrize("name,w_scale", [("mid", 12.0), ("head7b_small", 4.0)])
def test_proxy_top16_matches_oracle(name, w_scale):
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config(name, w_std=0.02 * w_scale)
    b = make_batch(cfg, device="cuda")
    hid, W = widen(cfg, b.hid_full), widen(cfg, b.W)
    N, k = len(b.tok_full), 16
    gamma = torch.empty(N, device="cuda")
    tidx = torch.empty(N, k, dtype=torch.int32, device="cuda")
    tprob = torch.empty(N, k, device="cuda")
    ws = torch.empty(B.ps_lmhead_score_proxy_workspace_size(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, k), dtype=torch.uint8,
                     device="cuda")
    B.ps_lmhead_score_proxy(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, b.dev["hid_full"], b.dev["W"], b.dev["tok_full"], gamma,
                            None, ws, k, tidx, tprob)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
    g_ref, _ = design.score_proxy(hid, W, b.tok_full)
    np.testing.assert_allclose(gamma.cpu().numpy(), g_ref, rtol=2e-4)
    ridx, rprob = design.topk_policy(hid, W, k)
    gi, gp = tidx.cpu().numpy(), tprob.cpu().numpy()
    z = hid @ W.T
    m = z.max(axis=1, keepdims=True)
    P = np.exp(z - m)
    P /= P.sum(axis=1, keepdims=True)
    rows = np.arange(N)[:, None]
    # the GPU's probabilities are those of its tokens, descending
    np.testing.assert_allclose(gp, P[rows, gi], rtol=2e-4, atol=1e-9)
    assert np.all(np.diff(gp, axis=1) <= 1e-7)
    # its set is a top-k set: same mass as the oracle's, and the same tokens away from near-ties
    np.testing.assert_allclose(P[rows, gi].sum(axis=1), rprob.sum(axis=1), rtol=1e-5)
    zk = np.sort(z, axis=1)[:, ::-1]
    clear = (zk[:, k - 1] - zk[:, k]) > 1e-3
    assert np.array_equal(np.sort(gi[clear], axis=1), np.sort(ridx[clear], axis=1))


@pytest.mark.parametrize("name", ["mid", "7b"])
def test_reward_uncertainty_matches_oracle(name):
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config(name)
    L = draw_lengths(cfg)
    N, k = int(L.sum()), 16
    rng = np.random.default_rng(2)
    # seeded top-16 lists over a small shared vocabulary so that completions overlap
    idx = np.stack([rng.choice(64, size=k, replace=False) for _ in range(N)]).astype(np.int32)
    prob = rng.dirichlet(np.ones(k + 1), size=N)[:, :k].astype(np.float32)
    R = (rng.random(cfg.B) < 0.5).astype(np.float32)
    R[:cfg.K] = 1.0                                   # one all-success group (u = 0 where all alive)
    T = int(L.max())
    u = torch.empty(cfg.P, T, device="cuda")
    ws = torch.empty(B.ps_reward_uncertainty_workspace_size(cfg.P, cfg.K), dtype=torch.uint8, device="cuda")
    B.ps_reward_uncertainty(cfg.P, cfg.K, T, torch.from_numpy(L).cuda(), torch.from_numpy(R).cuda(), k,
                            torch.from_numpy(idx).cuda(), torch.from_numpy(prob).cuda(), u, ws)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
    ref = design.reward_uncertainty(L, cfg.K, R, idx, prob)
    np.testing.assert_allclose(u.cpu().numpy(), ref, atol=2e-7)


def test_design_then_update_end_to_end():
    # proxy + top-16 -> u -> optimized design -> H = 0 sampling -> packing -> forward -> backward,
    # all on the device; every status clear and the outputs finite
    from paper_2606_29758_gb300 import _binding as B
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    D = b.dev
    N, T, k = b.total_len, b.T_max, 16
    gamma = torch.empty(N, device="cuda")
    tidx = torch.empty(N, k, dtype=torch.int32, device="cuda")
    tprob = torch.empty(N, k, device="cuda")
    ws_p = torch.empty(B.ps_lmhead_score_proxy_workspace_size(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, k),
                       dtype=torch.uint8, device="cuda")
    B.ps_lmhead_score_proxy(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, D["hid_full"], D["W"], D["tok_full"], gamma, None,
                            ws_p, k, tidx, tprob)
    u = torch.empty(cfg.P, T, device="cuda")
    ws_u = torch.empty(B.ps_reward_uncertainty_workspace_size(cfg.P, cfg.K), dtype=torch.uint8, device="cuda")
    B.ps_reward_uncertainty(cfg.P, cfg.K, T, D["L"], D["R"], k, tidx, tprob, u, ws_u)
    q = torch.empty(cfg.P, T, dtype=torch.int64, device="cuda")
    xi = torch.empty(cfg.P, T, dtype=torch.float64, device="cuda")
    ws_d = torch.empty(B.ps_design_cutoffs_workspace_size(cfg.P, cfg.K, T), dtype=torch.uint8, device="cuda")
    B.ps_design_cutoffs(cfg.P, cfg.K, T, D["L"], gamma, u, 40.0, B.PS_DESIGN_OPTIMIZED, 0.0, q, xi, ws_d)
    up = UpdatePass(PassShape(cfg.P, cfg.K, T, cfg.d, cfg.V, N), eps=cfg.eps, loss_scale=cfg.loss_scale,
                    mode=B.PS_MODE_TRUNC_ZERO)
    up.run(q, D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], 3, 0)
    torch.cuda.synchronize()
    for ws in (ws_p, ws_u, ws_d):
        assert B.ps_workspace_status(ws)[0] == B.PS_OK
    up.check_status()
    uu = u.cpu().numpy()
    assert np.all((uu >= 0) & (uu <= 0.5))
    x = xi.cpu().numpy()
    for p in range(cfg.P):
        Tp = int(b.L[p * cfg.K:(p + 1) * cfg.K].max())
        assert x[p, :Tp].sum() == pytest.approx(min(40.0, Tp), rel=1e-12)
    Nr = up.N
    assert torch.isfinite(up.loss).all() and torch.isfinite(up.dH[:Nr]).all() and torch.isfinite(up.dW).all()
    # weights are 1/xi of the realised distribution
    assert float(up.w[:Nr].min()) >= 1.0


def test_cutoff_design_holder_matches_the_abi_calls():
    # CutoffDesign runs the same three calls; its masses equal those of the calls made one by one
    from paper_2606_29758_gb300 import _binding as B
    from paper_2606_29758_gb300 import CutoffDesign, DesignShape
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    D = b.dev
    N, T, k = b.total_len, b.T_max, 16
    cd = CutoffDesign(DesignShape(cfg.P, cfg.K, T, cfg.d, cfg.V, N, k))
    q = cd.run(D["hid_full"], D["W"], D["tok_full"], D["L"], D["R"], 40.0).clone()
    gamma = torch.empty(N, device="cuda")
    tidx = torch.empty(N, k, dtype=torch.int32, device="cuda")
    tprob = torch.empty(N, k, device="cuda")
    ws_p = torch.zeros(B.ps_lmhead_score_proxy_workspace_size(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, k),
                       dtype=torch.uint8, device="cuda")
    B.ps_lmhead_score_proxy(N, cfg.d, cfg.V, B.PS_DTYPE_BF16, D["hid_full"], D["W"], D["tok_full"], gamma, None,
                            ws_p, k, tidx, tprob)
    u = torch.empty(cfg.P, T, device="cuda")
    ws_u = torch.zeros(B.ps_reward_uncertainty_workspace_size(cfg.P, cfg.K), dtype=torch.uint8, device="cuda")
    B.ps_reward_uncertainty(cfg.P, cfg.K, T, D["L"], D["R"], k, tidx, tprob, u, ws_u)
    q2 = torch.zeros(cfg.P, T, dtype=torch.int64, device="cuda")
    ws_d = torch.zeros(B.ps_design_cutoffs_workspace_size(cfg.P, cfg.K, T), dtype=torch.uint8, device="cuda")
    B.ps_design_cutoffs(cfg.P, cfg.K, T, D["L"], gamma, u, 40.0, B.PS_DESIGN_OPTIMIZED, 0.0, q2, None, ws_d)
    torch.cuda.synchronize()
    cd.check_status()
    assert torch.equal(q, q2) and torch.equal(cd.gamma, gamma) and torch.equal(cd.u, u)
    # the other strategies through the holder, checked against the oracle's masses
    for strategy, name, param in ((B.PS_DESIGN_UNIFORM, "uniform", 0.0), (B.PS_DESIGN_FIXED, "fixed", 12.0)):
        qs = cd.run(D["hid_full"], D["W"], D["tok_full"], D["L"], D["R"], 40.0, strategy, param).cpu().numpy()
        q_ref, _ = design.design_cutoff_masses(b.L, cfg.K, np.zeros(N, np.float32), None, 40.0, name, param=param)
        assert np.array_equal(qs.view(np.uint64), q_ref), name


def test_binarized_rewards_bit_exact_and_u_from_them():
    # Appendix G: labels y ~ Bernoulli(sigma(R)) equal the oracle's bit for bit (same Philox
    # stream, same fixed sigma sequence), and u_t from them matches the oracle's u_t
    from paper_2606_29758_gb300 import _binding as B
    from paper_2606_29758_gb300 import CutoffDesign, DesignShape
    rng = np.random.default_rng(8)
    R = np.concatenate([rng.normal(0.0, 2.0, 4000), [0.0, 40.0, -40.0, 60.0, -60.0, np.inf, -np.inf, np.nan],
                        rng.uniform(-0.01, 0.01, 88)]).astype(np.float32)
    Rd = torch.from_numpy(R).cuda()
    y = torch.empty_like(Rd)
    for seed, step, base in ((0, 0, 0), (7, 3, 0), (2**64 - 1, 2**40, 12345)):
        B.ps_binarize_rewards(len(R), Rd, seed, step, y, base)
        torch.cuda.synchronize()
        ref = design.binarize_rewards(R, seed, step, traj_base=base)
        assert np.array_equal(y.cpu().numpy(), ref), (seed, step)
    # u_t through CutoffDesign with continuous rewards: seeded top-16 lists over a small shared
    # vocabulary (as in the u_t test above) go into the holder's buffers, so both sides see the
    # same inputs
    cfg = get_config("mid")
    L = draw_lengths(cfg)
    N, k, T = int(L.sum()), 16, int(L.max())
    idx = np.stack([rng.choice(64, size=k, replace=False) for _ in range(N)]).astype(np.int32)
    prob = rng.dirichlet(np.ones(k + 1), size=N)[:, :k].astype(np.float32)
    Rc = rng.normal(0.0, 1.5, cfg.B).astype(np.float32)       # continuous rewards
    cd = CutoffDesign(DesignShape(cfg.P, cfg.K, T, cfg.d, cfg.V, N, k))
    cd.top_idx.copy_(torch.from_numpy(idx))
    cd.top_prob.copy_(torch.from_numpy(prob))
    cd.uncertainty(torch.from_numpy(L).cuda(), torch.from_numpy(Rc).cuda(), continuous=True, seed=4, step=1)
    torch.cuda.synchronize()
    cd.check_status()
    labels = design.binarize_rewards(Rc, 4, 1)
    assert np.array_equal(cd.y.cpu().numpy(), labels)
    u_ref = design.reward_uncertainty(L, cfg.K, labels, idx, prob)
    np.testing.assert_allclose(cd.u.cpu().numpy(), u_ref, atol=2e-7)


@pytest.mark.parametrize("name", ["7b", "long"])
def test_proxy_and_top16_at_full_size(name):
    # the launch configuration of the design stage in the benchmark: every rollout token of the
    # batch through the head (per-tile schedule without top-k, contiguous ranges with it); sampled
    # rows against the oracle, which evaluates them one by one
    from paper_2606_29758_gb300 import CutoffDesign, DesignShape
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    N, k = b.total_len, 16
    cd = CutoffDesign(DesignShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, N, k))
    cd.score(D["hid_full"], D["W"], D["tok_full"])
    g_topk, lp_topk = cd.gamma.clone(), cd.logp.clone()
    plain = CutoffDesign(DesignShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, N, 0))
    plain.score(D["hid_full"], D["W"], D["tok_full"])
    torch.cuda.synchronize()
    cd.check_status()
    plain.check_status()
    rng = np.random.default_rng(17)
    rows = np.unique(np.concatenate([rng.choice(N, 60, replace=False), [0, N - 1]]))
    from synthetic.generate import hidden_rows
    H = widen(cfg, hidden_rows(cfg, rows))
    W = widen(cfg, b.W)
    tok = b.tok_full[rows]
    g_ref, lp_ref = design.score_proxy(H, W, tok)
    sel = torch.from_numpy(rows).cuda()
    for g, lp in ((g_topk, lp_topk), (plain.gamma, plain.logp)):
        np.testing.assert_allclose(g[sel].cpu().numpy(), g_ref, rtol=2e-4)
        np.testing.assert_allclose(lp[sel].cpu().numpy(), lp_ref, rtol=1e-4, atol=2e-4)
    gi, gp = cd.top_idx[sel].cpu().numpy(), cd.top_prob[sel].cpu().numpy()
    z = H @ W.T
    P = np.exp(z - z.max(axis=1, keepdims=True))
    P /= P.sum(axis=1, keepdims=True)
    r = np.arange(len(rows))[:, None]
    np.testing.assert_allclose(gp, P[r, gi], rtol=2e-4, atol=1e-9)
    ridx, rprob = design.topk_policy(H, W, k)
    np.testing.assert_allclose(P[r, gi].sum(axis=1), rprob.sum(axis=1), rtol=1e-5)
    zk = np.sort(z, axis=1)[:, ::-1]
    clear = (zk[:, k - 1] - zk[:, k]) > 1e-3
    assert np.array_equal(np.sort(gi[clear], axis=1), np.sort(ridx[clear], axis=1))
