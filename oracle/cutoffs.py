"""Cutoff sampling and inverse-survival weights (oracle, float64 / exact integers).

Paper, Section 3.2: the cutoff H of a completion is random with survival
probabilities xi_t = Pr(H >= t | x), 1 >= xi_1 >= ... >= xi_T > 0. Only tokens
t <= H are back-propagated, and each retained token is reweighted by 1/xi_t
(Eq. truncated_update_Ghat; Algorithm 1, steps 10-11), which keeps the update
unbiased (Appendix B).

The cutoff distribution of prompt p is given as integer masses q_p[h], h = 1..T,
that sum to 2^62, so Pr(H = h) = q_p[h] / 2^62 exactly. With the cumulative sums
U_p[h] = q_p[1] + ... + q_p[h] (U_p[0] = 0), a uniform integer x on [0, 2^62)
selects H = min{h : x < U_p[h]}, and then
    xi_t = Pr(H >= t) = Pr(x >= U_p[t-1]) = (2^62 - U_p[t-1]) / 2^62 = S_p[t] / 2^62
holds exactly. The weight is w_p[t] = 1/xi_t = 2^62 / S_p[t].

In full mode (the untruncated control) H = L and every weight is 1.

In "trunc_zero" mode the masses may sum to less than 2^62: the deficit is Pr(H = 0) (no token of
the completion is kept; the design of Appendix F allows xi_1 < 1). Then H = 0 when x >= U[T], and
xi_t = (U[T] - U[t-1]) / 2^62.
"""
from __future__ import annotations

import numpy as np

from .philox import cutoff_uniform62

ONE62 = 1 << 62


def cumulative_masses(q_p: np.ndarray) -> np.ndarray:
    """U[h] for h = 0..T (U[0] = 0), as Python integers (exact)."""
    U = [0]
    for m in q_p:
        U.append(U[-1] + int(m))
    return U


def survival(q_p: np.ndarray):
    """S[t] = 2^62 - U[t-1] for t = 1..T (index t-1), exact integers."""
    U = cumulative_masses(q_p)
    return [ONE62 - U[t - 1] for t in range(1, len(q_p) + 1)]


def xi(q_p: np.ndarray) -> np.ndarray:
    """Survival probabilities xi_t = Pr(H >= t), t = 1..T, in float64."""
    return np.array([s / ONE62 for s in survival(q_p)], dtype=np.float64)


def survival_with_zero(q_p: np.ndarray):
    """Pr(H >= t) * 2^62 = U[T] - U[t-1] for t = 1..T (masses may leave Pr(H = 0) = the deficit)."""
    U = cumulative_masses(q_p)
    return [U[-1] - U[t - 1] for t in range(1, len(q_p) + 1)]


def inverse_survival_weights(q_p: np.ndarray, allow_zero: bool = False) -> np.ndarray:
    """w[t-1] = 1/xi_t = 2^62 / S[t] in float64 (+inf where S[t] = 0: never reached)."""
    out = np.empty(len(q_p), dtype=np.float64)
    S = survival_with_zero(q_p) if allow_zero else survival(q_p)
    for i, s in enumerate(S):
        out[i] = float(ONE62) / float(s) if s > 0 else np.inf
    return out


def cutoff_from_uniform(U, x: int, allow_zero: bool = False) -> int:
    """H = min{h >= 1 : x < U[h]} for x in [0, 2^62); 0 if x >= U[T] and allow_zero."""
    for h in range(1, len(U)):
        if x < U[h]:
            return h
    if allow_zero:
        return 0
    raise ValueError("masses do not cover x: they must sum to 2^62")


def sample_cutoffs(q: np.ndarray, L: np.ndarray, K: int, seed: int, step: int,
                   mode: str = "trunc", traj_base: int = 0):
    """Cutoffs H, prefix lengths n = min(H, L) and the weight table for B = len(L) trajectories.

    q: uint64 [P, T_max] masses; trajectory k belongs to prompt k // K; its random
    draw is keyed by the global index traj_base + k, so a sharded batch draws the
    same cutoffs as the whole batch.
    Returns (H int64 [B], n int64 [B], w_tab float64 [P, T_max]).
    """
    P, T_max = q.shape
    B = len(L)
    assert B == P * K
    H = np.zeros(B, dtype=np.int64)
    n = np.zeros(B, dtype=np.int64)
    if mode == "full":
        H[:] = L
        n[:] = L
        return H, n, np.ones((P, T_max), dtype=np.float64)
    zero = mode == "trunc_zero"
    w_tab = np.empty((P, T_max), dtype=np.float64)
    for p in range(P):
        U = cumulative_masses(q[p])
        if U[-1] > ONE62 or (U[-1] != ONE62 and not zero):
            raise ValueError(f"prompt {p}: masses sum to {U[-1]}, not 2^62")
        w_tab[p] = inverse_survival_weights(q[p], allow_zero=zero)
        for j in range(K):
            k = p * K + j
            x = cutoff_uniform62(seed, step, traj_base + k)
            H[k] = cutoff_from_uniform(U, x, allow_zero=zero)
            n[k] = min(int(H[k]), int(L[k]))
    return H, n, w_tab
