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
        if strategy != "uniform":
            continue


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
