"""Group-normalised advantages and ragged prefix packing (oracle).

Advantages (Section 3.1): critic-free methods broadcast one advantage over every
token of a completion, A = R - b(x), with b(x) the mean reward of the K
completions of the prompt (also Section 4, "The number of rollouts K"). The
group-normalised form additionally divides by the group's (population)
standard deviation plus 1e-6.

Packing (Algorithm 1, step 11): only tokens t <= H of completion k are updated,
so the update pass runs over the rows (k, t), k = 0..B-1, t = 1..n_k with
n_k = min(H_k, L_k), laid out back to back in that order. Row i = (k, t) takes
the completion's token t, its old log-probability and hidden state (source row
off_L[k] + t - 1 of the unpacked batch), the weight 1/xi_t of its prompt and the
advantage of its completion.
"""
from __future__ import annotations

import math

import numpy as np


def group_advantages(R: np.ndarray, K: int, adv_mode: int = 1) -> np.ndarray:
    """Per-completion advantage in float64; sums run sequentially over the group."""
    B = len(R)
    A = np.empty(B, dtype=np.float64)
    for p in range(B // K):
        r = [float(R[p * K + j]) for j in range(K)]
        s = 0.0
        for v in r:
            s += v
        mu = s / K
        if adv_mode == 0:
            for j in range(K):
                A[p * K + j] = r[j] - mu
            continue
        ss = 0.0
        for v in r:
            ss += (v - mu) * (v - mu)
        sigma = math.sqrt(ss / K)
        for j in range(K):
            A[p * K + j] = (r[j] - mu) / (sigma + 1e-6)
    return A


def pack_prefixes(L, n, K, w_tab, A, tok_full, oldlogp_full, hid_full=None):
    """Gather the packed prefix rows. Returns a dict of numpy arrays.

    cu_seqlens[k] = n_0 + ... + n_{k-1} (length B+1), and for each row i:
    src_row, row_traj (k), row_pos (t, 1-based), tok, oldlogp, w = w_tab[k // K][t-1],
    adv = A[k]; hid (if given) is hid_full[src_row].
    """
    B = len(L)
    off_L = np.zeros(B + 1, dtype=np.int64)
    cu = np.zeros(B + 1, dtype=np.int64)
    for k in range(B):
        off_L[k + 1] = off_L[k] + int(L[k])
        cu[k + 1] = cu[k] + int(n[k])
    N = int(cu[B])
    src = np.empty(N, dtype=np.int64)
    traj = np.empty(N, dtype=np.int64)
    pos = np.empty(N, dtype=np.int64)
    for k in range(B):
        t = np.arange(1, int(n[k]) + 1)
        src[cu[k]:cu[k + 1]] = off_L[k] + t - 1
        traj[cu[k]:cu[k + 1]] = k
        pos[cu[k]:cu[k + 1]] = t
    out = {
        "N": N,
        "cu_seqlens": cu,
        "src_row": src,
        "row_traj": traj,
        "row_pos": pos,
        "tok": np.asarray(tok_full)[src],
        "oldlogp": np.asarray(oldlogp_full, dtype=np.float64)[src],
        "w": np.asarray(w_tab)[traj // K, pos - 1],
        "adv": np.asarray(A)[traj],
    }
    if hid_full is not None:
        out["hid"] = np.asarray(hid_full)[src]
    return out
