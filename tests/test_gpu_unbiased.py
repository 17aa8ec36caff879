"""Unbiasedness of the CUDA path's truncated, reweighted update (Appendix B), by Monte Carlo.

The pass runs M times on one batch with M cutoff draws (Philox step counter 0..M-1); the mean of
its dW and of its hidden-state gradient must match the oracle's full-trajectory gradient within
the exact sampling error of the cutoffs. With per-token contributions g_t of one completion, the
variance of its reweighted sum is sum_{s,t} g_s g_t (1/xi_min(s,t) - 1) (Appendix C); it is
evaluated with suffix sums G_m = sum_{s >= m} g_s as sum_m (1/xi_m - 1) (G_m^2 - G_{m+1}^2).

The batch is the f32 Tiny workload (so dZ is not rounded to bf16) with a cutoff pmf that keeps
half its mass at T_p: every xi_t >= 1/2, the weights stay <= 2 and the Monte Carlo mean is close
to Gaussian. The same comparison against the mean a pass without the 1/xi weights would have
(a mistake planted in the oracle's reference) must fail by a wide margin.

The zero-cutoff mode runs the same check with masses that cover 3/4 of 2^62: the deficit is
Pr(H = 0) = 1/4 (a draw keeps no token of its completion, as an optimised design of Appendix F
allows), xi_t = Pr(H >= t) counts it (xi_1 = 3/4) and the weights are 1/xi_t of that distribution;
a reference whose weights ignore the deficit (xi_1 = 1) must fail as well.
"""
import numpy as np
import pytest

from oracle import lmhead
from oracle.cutoffs import ONE62, survival_with_zero, xi
from oracle.pack import group_advantages, pack_prefixes
from synthetic import get_config, make_batch

pytestmark = pytest.mark.gpu

M = 512


def _half_at_end_masses(L, K, T_max, zero=False):
    P = len(L) // K
    q = np.zeros((P, T_max), dtype=np.uint64)
    for p in range(P):
        T = int(L[p * K:(p + 1) * K].max())
        each = (1 << 61) // T
        q[p, :T] = each
        q[p, T - 1] += ONE62 - each * T
    if zero:
        q = (q // 4) * 3                        # Pr(H = 0) = 1/4 (up to 2^-62 per mass)
    return q


def _survival(q_p, zero):
    return np.array([v / ONE62 for v in survival_with_zero(q_p)]) if zero else xi(q_p)


def _oracle_full_and_variance(cfg, b, q, zero=False):
    """Full-trajectory dW and hidden-state gradient, the per-coordinate variance of one draw of the
    truncated estimator, and the means of two mistaken passes: one without the 1/xi weights, one
    whose weights take the masses as covering 2^62."""
    K = cfg.K
    L = b.L.astype(np.int64)
    A = group_advantages(b.R, K, cfg.adv_mode)
    pk = pack_prefixes(b.L, L, K, np.ones(q.shape), A, b.tok_full, b.oldlogp_full, b.hid_full)
    H = np.asarray(pk["hid"], dtype=np.float64)
    W = np.asarray(b.W, dtype=np.float64)
    f = lmhead.forward(H, W, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], cfg.eps, cfg.loss_scale)
    dH, dW = lmhead.backward(H, W, pk["tok"], f["lse"], f["coef"])
    dz = lmhead.dlogits(lmhead.logits(H, W), pk["tok"], f["lse"], f["coef"])
    var_w = np.zeros_like(dW)
    var_h = np.zeros_like(dH)
    for k in range(len(L)):
        x = _survival(q[k // K], zero)[:L[k]]  # t <= L_k <= T_p, so xi_t >= 1/2 (3/8 with a deficit)
        c = 1.0 / x - 1.0
        rows = np.nonzero(pk["row_traj"] == k)[0]
        rows = rows[np.argsort(pk["row_pos"][rows])]
        G = np.zeros_like(dW)
        prev = np.zeros_like(dW)
        for i in rows[::-1]:
            t = int(pk["row_pos"][i])
            G += np.outer(dz[i], H[i])
            sq = G * G
            var_w += c[t - 1] * (sq - prev)
            prev = sq
            var_h[pk["src_row"][i]] = c[t - 1] * dH[i] ** 2
    dhid = np.zeros((len(b.tok_full), cfg.d))
    dhid[pk["src_row"]] = dH
    # what the mean would be without the 1/xi weights: each token kept with probability xi_t
    idx = (pk["row_traj"] // K, pk["row_pos"] - 1)
    keep = np.stack([_survival(q_p, zero) for q_p in q])[idx]
    dW_unweighted = (keep[:, None] * dz).T @ H
    # weights 1/xi'_t with xi'_t = 1 - U[t-1]/2^62 (the deficit ignored): the mean is xi_t / xi'_t dz
    dW_wrong_xi = ((keep / np.stack([xi(q_p) for q_p in q])[idx])[:, None] * dz).T @ H
    return dW, dhid, var_w, var_h, dW_unweighted, dW_wrong_xi


@pytest.mark.parametrize("zero", [False, True], ids=["trunc", "trunc_zero"])
def test_monte_carlo_mean_of_the_cuda_pass_is_the_full_gradient(zero):
    import torch
    from paper_2606_29758_gb300 import PS_MODE_TRUNC, PS_MODE_TRUNC_ZERO, PassShape, UpdatePass
    cfg = get_config("tiny")
    b = make_batch(cfg, device="cuda")
    q = _half_at_end_masses(b.L, cfg.K, b.T_max, zero)
    D = dict(b.dev)
    D["q"] = torch.from_numpy(q.view(np.int64)).cuda()
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.float32),
                    eps=cfg.eps, loss_scale=cfg.loss_scale, adv_mode=cfg.adv_mode,
                    mode=PS_MODE_TRUNC_ZERO if zero else PS_MODE_TRUNC)
    acc_w = torch.zeros(cfg.V, cfg.d, dtype=torch.float64, device="cuda")
    acc_h = torch.zeros(b.total_len, cfg.d, dtype=torch.float64, device="cuda")
    kept = 0
    for step in range(M):
        N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], 5, step)
        acc_w += up.dW.double()
        acc_h.index_add_(0, up.src_row[:N].long(), up.dH[:N].double())
        kept += N
    torch.cuda.synchronize()
    up.check_status()
    mean_w = acc_w.cpu().numpy() / M
    mean_h = acc_h.cpu().numpy() / M

    dW, dhid, var_w, var_h, dW_unweighted, dW_wrong_xi = _oracle_full_and_variance(cfg, b, q, zero)
    assert kept < M * b.total_len          # the passes really truncated
    floor_w = (1e-6 * np.abs(dW).max()) ** 2
    floor_h = (1e-6 * np.abs(dhid).max()) ** 2
    z_w = (mean_w - dW) / np.sqrt(var_w / M + floor_w)
    z_h = (mean_h - dhid) / np.sqrt(var_h / M + floor_h)
    print("max |z| dW", np.abs(z_w).max(), "hidden", np.abs(z_h).max(), "kept", kept / (M * b.total_len))
    assert np.abs(z_w).max() < 6.0
    assert np.abs(z_h).max() < 6.0
    # the planted mistake: a reference without the inverse-survival weights is rejected
    z_bad = (mean_w - dW_unweighted) / np.sqrt(var_w / M + floor_w)
    assert np.abs(z_bad).max() > 12.0, np.abs(z_bad).max()
    if zero:
        z_bad = (mean_w - dW_wrong_xi) / np.sqrt(var_w / M + floor_w)
        assert np.abs(z_bad).max() > 12.0, np.abs(z_bad).max()
