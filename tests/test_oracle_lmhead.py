"""Pins for the oracle's LM-head loss and gradients (Eq. 1, Appendix D)."""
import math

import numpy as np
import pytest
from scipy.special import logsumexp as scipy_logsumexp

from oracle import lmhead


def _problem(N=7, d=5, V=11, seed=0, ratio_noise=0.05):
    rng = np.random.default_rng(seed)
    H = rng.standard_normal((N, d))
    W = rng.standard_normal((V, d)) * 0.3
    tok = rng.integers(0, V, N)
    z = H @ W.T
    logp = z[np.arange(N), tok] - scipy_logsumexp(z, axis=1)
    old = logp + rng.standard_normal(N) * ratio_noise
    adv = rng.choice([-1.3, -0.4, 0.7, 1.1], N)
    w = rng.uniform(1.0, 4.0, N)
    return H, W, tok, old, adv, w


def _loss(H, W, tok, old, adv, w, eps, c):
    return lmhead.forward(H, W, tok, old, adv, w, eps, c)["loss"]


def test_lse_matches_scipy():
    rng = np.random.default_rng(1)
    z = rng.standard_normal((9, 300)) * 20
    np.testing.assert_allclose(lmhead.logsumexp_rows(z), scipy_logsumexp(z, axis=1), rtol=1e-14)


def test_uniform_head_gives_log_uniform():
    # identical vocabulary rows => uniform softmax => logp = -log V exactly (up to rounding)
    V, d = 37, 4
    W = np.tile(np.arange(1.0, d + 1)[None], (V, 1))
    H = np.random.default_rng(0).standard_normal((3, d))
    f = lmhead.forward(H, W, np.array([0, 5, 36]), np.zeros(3), np.ones(3), np.ones(3), 0.2, 1.0)
    np.testing.assert_allclose(f["logp"], -math.log(V), rtol=1e-13)


def test_surrogate_textbook_cases():
    eps = 0.2
    # ratio 1: surrogate = A; clip never binds
    assert lmhead.clipped_surrogate(1.0, 2.0, eps) == 2.0
    # A > 0, r > 1+eps: clipped value (1+eps) A, gradient zero
    assert lmhead.clipped_surrogate(1.5, 2.0, eps) == pytest.approx(2.4)
    assert lmhead.clip_binding(1.5, 2.0, eps)
    # A > 0, r < 1-eps: min picks r A (pessimistic), gradient flows
    assert lmhead.clipped_surrogate(0.5, 2.0, eps) == pytest.approx(1.0)
    assert not lmhead.clip_binding(0.5, 2.0, eps)
    # A < 0, r < 1-eps: clipped value (1-eps) A, gradient zero
    assert lmhead.clipped_surrogate(0.5, -2.0, eps) == pytest.approx(-1.6)
    assert lmhead.clip_binding(0.5, -2.0, eps)
    # A < 0, r > 1+eps: r A, gradient flows
    assert lmhead.clipped_surrogate(1.5, -2.0, eps) == pytest.approx(-3.0)
    assert not lmhead.clip_binding(1.5, -2.0, eps)


def test_ratio_one_and_no_clip_reduce_to_policy_gradient():
    H, W, tok, old, adv, w = _problem()
    f0 = lmhead.forward(H, W, tok, old, adv, w, 0.2, 0.5)
    # old = current logp => r = 1 => loss = -c sum w A, coef = -c w A
    g = lmhead.forward(H, W, tok, f0["logp"], adv, w, 0.2, 0.5)
    np.testing.assert_allclose(g["ratio"], 1.0, rtol=1e-15)
    assert g["loss"] == pytest.approx(-0.5 * float(np.sum(w * adv)), rel=1e-14)
    np.testing.assert_allclose(g["coef"], -0.5 * w * adv, rtol=1e-14)
    # eps -> infinity: coef = -c w A r for every row (plain importance-weighted gradient)
    h = lmhead.forward(H, W, tok, old, adv, w, 1e9, 0.5)
    np.testing.assert_allclose(h["coef"], -0.5 * w * adv * h["ratio"], rtol=1e-14)


@pytest.mark.parametrize("noise", [0.05, 0.6])
def test_gradients_match_central_differences(noise):
    eps, c = 0.2, 0.25
    H, W, tok, old, adv, w = _problem(seed=3, ratio_noise=noise)
    f = lmhead.forward(H, W, tok, old, adv, w, eps, c)
    # keep rows away from the clip kinks so the loss is smooth around the point
    kink = np.minimum(np.abs(f["ratio"] - (1 + eps)), np.abs(f["ratio"] - (1 - eps)))
    keep = kink > 1e-3
    H, tok, old, adv, w = H[keep], tok[keep], old[keep], adv[keep], w[keep]
    f = lmhead.forward(H, W, tok, old, adv, w, eps, c)
    dH, dW = lmhead.backward(H, W, tok, f["lse"], f["coef"])
    h = 1e-6
    for (i, j) in [(0, 0), (1, 3), (H.shape[0] - 1, 4)]:
        Hp, Hm = H.copy(), H.copy()
        Hp[i, j] += h
        Hm[i, j] -= h
        fd = (_loss(Hp, W, tok, old, adv, w, eps, c) - _loss(Hm, W, tok, old, adv, w, eps, c)) / (2 * h)
        assert dH[i, j] == pytest.approx(fd, rel=1e-6, abs=1e-10)
    for (v, j) in [(0, 0), (int(tok[0]), 2), (10, 4)]:
        Wp, Wm = W.copy(), W.copy()
        Wp[v, j] += h
        Wm[v, j] -= h
        fd = (_loss(H, Wp, tok, old, adv, w, eps, c) - _loss(H, Wm, tok, old, adv, w, eps, c)) / (2 * h)
        assert dW[v, j] == pytest.approx(fd, rel=1e-6, abs=1e-10)
    # logp gradient: coef = d loss / d logp, checked through the old log-prob (d/d old = -coef)
    for i in range(min(3, len(tok))):
        op, om = old.copy(), old.copy()
        op[i] += h
        om[i] -= h
        fd = (_loss(H, W, tok, op, adv, w, eps, c) - _loss(H, W, tok, om, adv, w, eps, c)) / (2 * h)
        assert -f["coef"][i] == pytest.approx(fd, rel=1e-6, abs=1e-10)


def test_vocab_sum_of_dW_vanishes():
    # sum_v (e_o - p)_v = 0 for every row, so sum_v dW[v, :] = 0 and sum_v dZ[i, v] = 0
    H, W, tok, old, adv, w = _problem(N=20, d=6, V=50, seed=5)
    f = lmhead.forward(H, W, tok, old, adv, w, 0.2, 1.0)
    _, dW = lmhead.backward(H, W, tok, f["lse"], f["coef"])
    assert np.abs(dW.sum(axis=0)).max() < 1e-13 * np.abs(dW).max() * W.shape[0]
    z = lmhead.logits(H, W)
    dz = lmhead.dlogits(z, tok, f["lse"], f["coef"])
    assert np.abs(dz.sum(axis=1)).max() < 1e-14


def test_subsets_match_full_evaluation():
    H, W, tok, old, adv, w = _problem(N=30, d=6, V=40, seed=8)
    f = lmhead.forward(H, W, tok, old, adv, w, 0.2, 1.0)
    rows = np.array([3, 0, 29, 17])
    g = lmhead.forward(H, W, tok, old, adv, w, 0.2, 1.0, rows=rows)
    for k in ("lse", "logp", "ratio", "coef", "row_loss"):
        np.testing.assert_allclose(g[k], f[k][rows], rtol=1e-14)
    dH, dW = lmhead.backward(H, W, tok, f["lse"], f["coef"])
    sH, sW = lmhead.backward(H, W, tok, f["lse"], f["coef"], dh_rows=rows, dw_vocab=np.array([1, 39, int(tok[0])]))
    np.testing.assert_allclose(sH, dH[rows], rtol=1e-12, atol=1e-16)
    np.testing.assert_allclose(sW, dW[[1, 39, int(tok[0])]], rtol=1e-12, atol=1e-16)


def test_brute_force_single_row():
    # d = 1, V = 2: logp of token 0 is -log(1 + exp(z1 - z0)) with z = W h
    H = np.array([[0.7]])
    W = np.array([[1.5], [-0.25]])
    f = lmhead.forward(H, W, np.array([0]), np.array([-0.1]), np.array([1.0]), np.array([2.0]), 0.2, 1.0)
    z0, z1 = 1.5 * 0.7, -0.25 * 0.7
    lp = -math.log1p(math.exp(z1 - z0))
    assert f["logp"][0] == pytest.approx(lp, rel=1e-15)
    r = math.exp(lp + 0.1)
    assert f["loss"] == pytest.approx(-2.0 * min(r, min(max(r, 0.8), 1.2)), rel=1e-15)
