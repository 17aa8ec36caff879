"""The whole update pass in the oracle, in the paper's order (Algorithm 1, steps 6 and 10-11):
advantages -> cutoffs -> packed prefixes -> clipped surrogate loss -> head gradients.
"""
from __future__ import annotations

import numpy as np

from .cutoffs import sample_cutoffs
from .lmhead import backward, forward
from .pack import group_advantages, pack_prefixes


def run(q, L, K, R, tok_full, oldlogp_full, hid_full, W, eps, loss_scale, seed, step,
        mode="trunc", adv_mode=1, traj_base=0, grads=True):
    """hid_full and W are float arrays (bf16 inputs already widened exactly)."""
    H, n, w_tab = sample_cutoffs(q, L, K, seed, step, mode=mode, traj_base=traj_base)
    A = group_advantages(R, K, adv_mode)
    pk = pack_prefixes(L, n, K, w_tab, A, tok_full, oldlogp_full, hid_full)
    fw = forward(pk["hid"], W, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], eps, loss_scale)
    out = {"H": H, "n": n, "w_tab": w_tab, "A": A, "pack": pk, "fwd": fw}
    if grads:
        out["dH"], out["dW"] = backward(pk["hid"], W, pk["tok"], fw["lse"], fw["coef"])
    return out


def widen(cfg, m: np.ndarray) -> np.ndarray:
    """bf16 bits (uint16) or float32 -> float64, exactly."""
    if m.dtype == np.uint16:
        return (m.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return np.asarray(m, dtype=np.float64)
