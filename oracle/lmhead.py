"""LM-head clipped-surrogate loss and its gradients (oracle, float64).

For a packed row i with hidden state h_i, chosen token o_i, old log-probability
l_i, advantage A_i and weight w_i = 1/xi_t:

  logits        z_i = W h_i, W stored [V, d] (Appendix D: z = W h + b; no bias here)
  log-prob      logp_i = z_{i,o_i} - log sum_v exp(z_{i,v})
  ratio         r_i = pi_theta / pi_old = exp(logp_i - l_i)             (Section 3.1)
  surrogate     s_i = min(r_i A_i, clip(r_i, 1-eps, 1+eps) A_i)          (Eq. 1)
  loss          loss = -c sum_i w_i s_i, c = 1/(P K)                     (Eq. truncated_update_Ghat:
                1/K per prompt, seq-sum over retained tokens, averaged over P prompts;
                the minus sign turns the maximised objective into a loss)

Gradient. The surrogate follows r A unless the clip is binding, i.e. unless
(A > 0 and r > 1+eps) or (A < 0 and r < 1-eps), where it is constant. So
  coef_i = d loss / d logp_i = -c w_i A_i r_i  (0 where the clip binds).
Appendix D gives the softmax-head score d logp / dz = e_o - p, hence
  dZ_{i,v} = coef_i (1[v = o_i] - p_{i,v}),  p_{i,v} = exp(z_{i,v} - lse_i),
  dH = dZ W   ([N, d]),   dW = dZ^T H   ([V, d], same storage as W).
"""
from __future__ import annotations

import math

import numpy as np

ROW_BLOCK = 128


def logits(Hrows: np.ndarray, W: np.ndarray) -> np.ndarray:
    return np.asarray(Hrows, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T


def logsumexp_rows(z: np.ndarray) -> np.ndarray:
    """log sum_v exp(z_v) per row, shifted by the row maximum for range safety."""
    m = z.max(axis=1)
    return m + np.log(np.exp(z - m[:, None]).sum(axis=1))


def clipped_surrogate(r, A, eps):
    """min(r A, clip(r, 1-eps, 1+eps) A), Eq. 1 (per token)."""
    r = np.asarray(r, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    return np.minimum(r * A, np.clip(r, 1.0 - eps, 1.0 + eps) * A)


def clip_binding(r, A, eps):
    """True where the clipped branch is the minimum and its slope in r is zero."""
    r = np.asarray(r, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    return ((A > 0) & (r > 1.0 + eps)) | ((A < 0) & (r < 1.0 - eps))


def forward(H, W, tok, oldlogp, adv, w, eps, loss_scale, rows=None):
    """Per-row lse, logp, ratio, row_loss, coef (float64) and the total loss.

    rows: optional subset of row indices (all outputs are then for that subset and
    `loss` is the subset's sum).
    """
    idx = np.arange(len(tok)) if rows is None else np.asarray(rows, dtype=np.int64)
    W64 = np.asarray(W, dtype=np.float64)
    lse = np.empty(idx.size)
    zt = np.empty(idx.size)
    for b0 in range(0, idx.size, ROW_BLOCK):
        sel = idx[b0:b0 + ROW_BLOCK]
        z = logits(np.asarray(H)[sel], W64)
        lse[b0:b0 + sel.size] = logsumexp_rows(z)
        zt[b0:b0 + sel.size] = z[np.arange(sel.size), np.asarray(tok)[sel]]
    logp = zt - lse
    A = np.asarray(adv, dtype=np.float64)[idx]
    wt = np.asarray(w, dtype=np.float64)[idx]
    ratio = np.exp(logp - np.asarray(oldlogp, dtype=np.float64)[idx])
    s = clipped_surrogate(ratio, A, eps)
    row_loss = -loss_scale * wt * s
    coef = np.where(clip_binding(ratio, A, eps), 0.0, -loss_scale * wt * A * ratio)
    return {
        "rows": idx, "lse": lse, "logp": logp, "ratio": ratio, "row_loss": row_loss,
        "coef": coef, "loss": math.fsum(row_loss.tolist()),
    }


def dlogits(z: np.ndarray, tok_rows: np.ndarray, lse_rows: np.ndarray, coef_rows: np.ndarray) -> np.ndarray:
    """dZ = coef (onehot(o) - softmax(z)) for a block of rows (Appendix D score, chain rule)."""
    dz = -np.exp(z - lse_rows[:, None])
    dz[np.arange(z.shape[0]), tok_rows] += 1.0
    return coef_rows[:, None] * dz


def backward(H, W, tok, lse, coef, dh_rows=None, dw_vocab=None):
    """dH (rows dh_rows, default all) and dW (vocab rows dw_vocab, default all), float64.

    lse and coef must cover all N rows (dW sums over every row).
    """
    H = np.asarray(H)
    W64 = np.asarray(W, dtype=np.float64)
    N = len(tok)
    tok = np.asarray(tok)
    hr = np.arange(N) if dh_rows is None else np.asarray(dh_rows, dtype=np.int64)
    vr = np.arange(W64.shape[0]) if dw_vocab is None else np.asarray(dw_vocab, dtype=np.int64)
    dH = np.empty((hr.size, W64.shape[1]))
    for b0 in range(0, hr.size, ROW_BLOCK):
        sel = hr[b0:b0 + ROW_BLOCK]
        z = logits(H[sel], W64)
        dH[b0:b0 + sel.size] = dlogits(z, tok[sel], lse[sel], coef[sel]) @ W64
    dW = np.zeros((vr.size, W64.shape[1]))
    Wv = W64[vr]
    for b0 in range(0, N, ROW_BLOCK):
        sel = np.arange(b0, min(N, b0 + ROW_BLOCK))
        Hb = np.asarray(H[sel], dtype=np.float64)
        z = Hb @ Wv.T
        dz = -np.exp(z - lse[sel][:, None])
        hit = tok[sel][:, None] == vr[None, :]
        dz[hit] += 1.0
        dW += (coef[sel][:, None] * dz).T @ Hb
    return dH, dW
