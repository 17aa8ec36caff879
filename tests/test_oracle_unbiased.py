"""Unbiasedness of the truncated, reweighted update (Appendix B), pinned two ways:
exact enumeration over every cutoff combination, and Monte Carlo over seeds
with the exact cutoff-induced variance as the tolerance."""
import itertools

import numpy as np
import pytest

from oracle import lmhead
from oracle.cutoffs import ONE62, cumulative_masses, inverse_survival_weights, sample_cutoffs, xi
from oracle.pack import group_advantages, pack_prefixes
from synthetic.generate import beta_masses


def _setup(seed=0, L=(6, 9), d=4, V=13):
    rng = np.random.default_rng(seed)
    L = np.array(L, dtype=np.int32)
    K = len(L)
    T = int(L.max())
    total = int(L.sum())
    q = beta_masses(T, 1.3, 2.2)[None]
    hid = rng.standard_normal((total, d))
    W = rng.standard_normal((V, d)) * 0.4
    tok = rng.integers(0, V, total)
    old = rng.standard_normal(total) * 0.3 - 2.0
    R = np.array([1.0, 0.0] + [float(i % 2) for i in range(K - 2)], dtype=np.float32)
    return dict(L=L, K=K, q=q, hid=hid, W=W, tok=tok, old=old, R=R, c=1.0 / K, eps=0.2)


def _grads_for_cutoffs(s, H, mode="trunc", w_tab=None):
    """Gradients w.r.t. W and w.r.t. the unpacked hidden states for given cutoffs (H = 0 keeps no
    token of its completion); w_tab overrides the weights 1/xi_t of the masses."""
    L = s["L"]
    n = np.minimum(H, L) if mode == "trunc" else L.astype(np.int64)
    if w_tab is None:
        w_tab = inverse_survival_weights(s["q"][0])[None] if mode == "trunc" else np.ones_like(s["q"], dtype=np.float64)
    if n.sum() == 0:
        return np.zeros_like(s["W"]), np.zeros_like(s["hid"])
    A = group_advantages(s["R"], s["K"], 1)
    pk = pack_prefixes(L, n, s["K"], w_tab, A, s["tok"], s["old"], s["hid"])
    f = lmhead.forward(pk["hid"], s["W"], pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], s["eps"], s["c"])
    dH, dW = lmhead.backward(pk["hid"], s["W"], pk["tok"], f["lse"], f["coef"])
    dhid = np.zeros_like(s["hid"])
    dhid[pk["src_row"]] = dH
    return dW, dhid


def test_exact_enumeration_equals_full_update():
    s = _setup()
    T = int(s["L"].max())
    p = np.array([int(m) / ONE62 for m in s["q"][0]])
    EW = 0.0
    Ehid = 0.0
    for hs in itertools.product(range(1, T + 1), repeat=s["K"]):
        pr = float(np.prod([p[h - 1] for h in hs]))
        if pr == 0.0:
            continue
        dW, dhid = _grads_for_cutoffs(s, np.array(hs))
        EW = EW + pr * dW
        Ehid = Ehid + pr * dhid
    GW, Ghid = _grads_for_cutoffs(s, None, mode="full")
    np.testing.assert_allclose(EW, GW, rtol=1e-11, atol=1e-13 * np.abs(GW).max())
    np.testing.assert_allclose(Ehid, Ghid, rtol=1e-11, atol=1e-13 * np.abs(Ghid).max())


def test_off_by_one_weight_would_be_biased():
    # the same enumeration with weights shifted by one position is visibly biased
    s = _setup(seed=2)
    T = int(s["L"].max())
    p = np.array([int(m) / ONE62 for m in s["q"][0]])
    w_good = inverse_survival_weights(s["q"][0])
    w_bad = np.concatenate([w_good[1:], w_good[-1:]])
    A = group_advantages(s["R"], s["K"], 1)
    GW, _ = _grads_for_cutoffs(s, None, mode="full")
    EW = 0.0
    for hs in itertools.product(range(1, T + 1), repeat=s["K"]):
        pr = float(np.prod([p[h - 1] for h in hs]))
        n = np.minimum(np.array(hs), s["L"])
        pk = pack_prefixes(s["L"], n, s["K"], w_bad[None], A, s["tok"], s["old"], s["hid"])
        f = lmhead.forward(pk["hid"], s["W"], pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], s["eps"], s["c"])
        EW = EW + pr * lmhead.backward(pk["hid"], s["W"], pk["tok"], f["lse"], f["coef"])[1]
    assert np.abs(EW - GW).max() > 1e-3 * np.abs(GW).max()


@pytest.mark.slow
def test_monte_carlo_mean_within_exact_sampling_error():
    s = _setup(seed=4, L=(14, 20, 9, 17), d=3, V=7)
    T = int(s["L"].max())
    M = 600
    acc = 0.0
    L = s["L"]
    for step in range(M):
        H, _, _ = sample_cutoffs(s["q"], L, s["K"], seed=77, step=step)
        acc = acc + _grads_for_cutoffs(s, H)[0]
    mean = acc / M
    GW, _ = _grads_for_cutoffs(s, None, mode="full")
    # exact variance: per trajectory Var = sum_{s,t} g_s g_t (1/xi_min(s,t) - 1)
    x = xi(s["q"][0])
    A = group_advantages(s["R"], s["K"], 1)
    pk = pack_prefixes(L, L.astype(np.int64), s["K"], np.ones((1, T)), A, s["tok"], s["old"], s["hid"])
    f = lmhead.forward(pk["hid"], s["W"], pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], s["eps"], s["c"])
    z = lmhead.logits(pk["hid"], s["W"])
    dz = lmhead.dlogits(z, pk["tok"], f["lse"], f["coef"])
    var = np.zeros_like(GW)
    for k in range(s["K"]):
        rows = np.nonzero(pk["row_traj"] == k)[0]
        g = np.stack([np.outer(dz[i], pk["hid"][i]) for i in rows])          # [n_k, V, d]
        t = pk["row_pos"][rows]
        C = 1.0 / x[np.minimum.outer(t, t) - 1] - 1.0                         # [n_k, n_k]
        var += np.einsum("svd,st,tvd->vd", g, C, g)
    zscore = (mean - GW) / np.sqrt(var / M + 1e-300)
    assert np.abs(zscore).max() < 4.5
    assert np.abs(mean - GW).max() > 0  # the estimate is random, not the full update itself


def _deficit_setup():
    # masses summing to 3/4 of 2^62: the deficit, Pr(H = 0) = 1/4, keeps no token of a completion
    # (the zero-cutoff sampling of an optimised design, Appendix F, where xi_1 < 1)
    s = _setup(seed=5, L=(5, 8))
    s["q"] = (s["q"] // 4) * 3
    return s


def _enumerate_with_zero(s, w_tab):
    T = int(s["L"].max())
    U = cumulative_masses(s["q"][0])
    p = [(ONE62 - U[-1]) / ONE62] + [int(m) / ONE62 for m in s["q"][0]]      # h = 0, 1, ..., T
    EW, Ehid = 0.0, 0.0
    for hs in itertools.product(range(T + 1), repeat=s["K"]):
        pr = float(np.prod([p[h] for h in hs]))
        dW, dhid = _grads_for_cutoffs(s, np.array(hs), w_tab=w_tab)
        EW = EW + pr * dW
        Ehid = Ehid + pr * dhid
    return EW, Ehid


def test_exact_enumeration_with_zero_cutoffs_equals_full_update():
    s = _deficit_setup()
    assert 0.24 < (ONE62 - cumulative_masses(s["q"][0])[-1]) / ONE62 < 0.26
    w = inverse_survival_weights(s["q"][0], allow_zero=True)
    assert w[0] == pytest.approx(ONE62 / float(cumulative_masses(s["q"][0])[-1]), rel=1e-15)   # 1/xi_1 = 4/3
    EW, Ehid = _enumerate_with_zero(s, w[None])
    GW, Ghid = _grads_for_cutoffs(s, None, mode="full")
    np.testing.assert_allclose(EW, GW, rtol=1e-11, atol=1e-13 * np.abs(GW).max())
    np.testing.assert_allclose(Ehid, Ghid, rtol=1e-11, atol=1e-13 * np.abs(Ghid).max())
    # planted mistake: weights taken as if the masses covered 2^62 (xi_1 = 1) leave the mean biased
    w_bad = np.array([ONE62 / float(ONE62 - u) for u in cumulative_masses(s["q"][0])[:-1]])
    EW_bad, _ = _enumerate_with_zero(s, w_bad[None])
    assert np.abs(EW_bad - GW).max() > 0.1 * np.abs(GW).max()
