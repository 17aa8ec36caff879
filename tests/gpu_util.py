"""Helpers for the GPU parity tests: run the CUDA pass through the C ABI and the oracle on
the same seeded inputs, and compare."""
from __future__ import annotations

import numpy as np

from oracle import lmhead
from oracle.cutoffs import sample_cutoffs
from oracle.pack import group_advantages, pack_prefixes
from oracle.pipeline import widen
from synthetic import make_batch

# Tolerances (stated for the path): cutoffs and indices bit-exact; loss 1e-3 relative;
# dH and dW 2e-2 max-relative (max |gpu - ref| / max |ref|) against the oracle on the
# rounded inputs.
LOSS_RTOL = 1e-3
GRAD_MAXREL = 2e-2


def gpu_pass(cfg, batch=None, chunk_rows=32768, grads=True, seed=None, step=None):
    import torch
    from paper_2606_29758_gb300 import PS_MODE_FULL, PS_MODE_TRUNC, PassShape, UpdatePass
    b = batch if batch is not None else make_batch(cfg, device="cuda")
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    shape = PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, dt, chunk_rows)
    up = UpdatePass(shape, eps=cfg.eps, loss_scale=cfg.loss_scale,
                    mode=PS_MODE_FULL if cfg.mode == "full" else PS_MODE_TRUNC, adv_mode=cfg.adv_mode)
    D = b.dev
    up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"],
           cfg.seed if seed is None else seed, cfg.step if step is None else step, grads=grads)
    torch.cuda.synchronize()
    up.check_status()
    return b, up


def to_np(up, N):
    import torch
    out = {k: getattr(up, k).cpu().numpy() for k in ("H", "n", "w_tab", "cu_seqlens")}
    for k in ("src_row", "row_traj", "row_pos", "tok", "oldlogp", "w", "adv", "lse", "logp", "ratio", "coef",
              "row_loss", "dH"):
        out[k] = getattr(up, k)[:N].cpu().numpy()
    h = up.hid[:N]
    out["hid"] = (h.view(torch.int16).cpu().numpy().view(np.uint16) if h.dtype == torch.bfloat16
                  else h.cpu().numpy())
    out["dW"] = up.dW.cpu().numpy()
    out["loss"] = float(up.loss.item())
    return out


def oracle_prefix(cfg, b, seed=None, step=None):
    """Oracle cutoffs, advantages and packing (no head)."""
    mode = "full" if cfg.mode == "full" else "trunc"
    H, n, w_tab = sample_cutoffs(b.q, b.L, cfg.K, cfg.seed if seed is None else seed,
                                 cfg.step if step is None else step, mode=mode)
    A = group_advantages(b.R, cfg.K, cfg.adv_mode)
    pk = pack_prefixes(b.L, n, cfg.K, w_tab, A, b.tok_full, b.oldlogp_full, b.hid_full)
    return H, n, w_tab, A, pk


def check_prefix(cfg, b, g, seed=None, step=None):
    H, n, w_tab, A, pk = oracle_prefix(cfg, b, seed, step)
    N = pk["N"]
    assert np.array_equal(g["H"], H), "cutoffs differ"
    assert np.array_equal(g["n"], n)
    ref_w = w_tab.astype(np.float32)
    fin = np.isfinite(ref_w)
    assert np.array_equal(g["w_tab"][fin], ref_w[fin])
    assert np.all(np.isinf(g["w_tab"][~fin]))
    assert np.array_equal(g["cu_seqlens"], pk["cu_seqlens"])
    for k in ("src_row", "row_traj", "row_pos", "tok"):
        assert np.array_equal(g[k], pk[k]), k
    assert np.array_equal(g["oldlogp"], pk["oldlogp"].astype(np.float32))
    assert np.array_equal(g["w"], pk["w"].astype(np.float32))
    assert np.array_equal(g["adv"], pk["adv"].astype(np.float32))
    assert np.array_equal(g["hid"], pk["hid"])
    return N, pk


def maxrel(a, b):
    den = np.abs(b).max()
    return float(np.abs(a - b).max() / den) if den > 0 else float(np.abs(a - b).max())


def check_head(cfg, b, g, pk, rows=None, grads=True, report=None):
    """Compare the head outputs with the oracle. rows: subset of packed rows (None = all)."""
    W = widen(cfg, b.W)
    H = widen(cfg, pk["hid"])
    f = lmhead.forward(H, W, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], cfg.eps, cfg.loss_scale, rows=rows)
    idx = f["rows"]
    lse_err = float(np.abs(g["lse"][idx] - f["lse"]).max())
    logp_err = float(np.abs(g["logp"][idx] - f["logp"]).max())
    ratio_err = float((np.abs(g["ratio"][idx] - f["ratio"]) / f["ratio"]).max())
    near = np.minimum(np.abs(f["ratio"] - (1 + cfg.eps)), np.abs(f["ratio"] - (1 - cfg.eps))) < 1e-5
    cref = f["coef"][~near]
    coef_err = maxrel(g["coef"][idx][~near], cref) if cref.size else 0.0
    rl_err = maxrel(g["row_loss"][idx], f["row_loss"])
    stats = dict(lse=lse_err, logp=logp_err, ratio=ratio_err, coef=coef_err, row_loss=rl_err, near_clip=int(near.sum()))
    assert lse_err < 2e-4, stats
    assert logp_err < 2e-4, stats
    assert ratio_err < 2e-4, stats
    assert coef_err < 2e-4, stats
    assert rl_err < 2e-4, stats
    if rows is None:
        rel = abs(g["loss"] - f["loss"]) / max(abs(f["loss"]), 1e-300)
        stats["loss_rel"] = rel
        assert rel < LOSS_RTOL, stats
    if grads:
        # the oracle's backward uses its own lse and coef
        if rows is None:
            dH, dW = lmhead.backward(H, W, pk["tok"], f["lse"], f["coef"])
            stats["dH"] = maxrel(g["dH"], dH)
            stats["dW"] = maxrel(g["dW"], dW)
        else:
            lse_o = np.zeros(len(pk["tok"]))
            coef_o = np.zeros(len(pk["tok"]))
            lse_o[idx], coef_o[idx] = f["lse"], f["coef"]     # oracle values; only these rows are read
            dH, _ = lmhead.backward(H, W, pk["tok"], lse_o, coef_o, dh_rows=idx, dw_vocab=[])
            stats["dH"] = maxrel(g["dH"][idx], dH)
        assert stats["dH"] < GRAD_MAXREL, stats
        if "dW" in stats:
            assert stats["dW"] < GRAD_MAXREL, stats
    if report is not None:
        report.update(stats)
        report["oracle_rows"], report["oracle_lse"], report["oracle_coef"] = idx, f["lse"], f["coef"]
    return stats

