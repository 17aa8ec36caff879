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


# ----------------------------------------------------------------------------- the launch schedule
# The library's row schedule, restated so that a parity check can touch every place where a
# launch changes hands: the backward's chunking (csrc/psppo_api.cu) and the row bands of the
# forward, recompute and dH/dW GEMMs (csrc/lmhead_bf16.cu).
FWD_BAND_L2_BYTES = 30e6      # hidden rows of one forward band
REC_BAND_BLOCKS = 32          # 128-row blocks per recompute band
GRAD_BAND_ROWS = 4 * 256      # dH / dW bands: 4 tiles of 256 rows


def bwd_chunks(N, ws_chunk_rows):
    """[r0, r1) of every backward chunk: as few as a workspace of ws_chunk_rows holds, of equal
    size rounded up to 128 rows."""
    chunk = ws_chunk_rows // 128 * 128
    nch = -(-N // chunk)
    chunk = -(-(-(-N // nch)) // 128) * 128
    chunk = min(chunk, N)
    return [(r0, min(N, r0 + chunk)) for r0 in range(0, N, chunk)]


def schedule_rows(cfg, N, ws_chunk_rows, seed=1234):
    """One row of every 128-row block (seeded), and the rows on both sides of every forward band
    edge, backward chunk edge, recompute band edge, dH/dW band edge, plus the last row."""
    rng = np.random.default_rng(seed)
    starts = np.arange(0, N, 128)
    rows = set((starts + rng.integers(0, np.minimum(128, N - starts))).tolist())

    def edge(e):
        rows.update(r for r in (e - 1, e) if 0 <= r < N)

    tile = 128 * (2 if cfg.d >= 1024 else 1)          # the forward's tile height at this d
    band = max(1, int(FWD_BAND_L2_BYTES // (tile * cfg.d * 2)))
    for e in range(0, N, band * tile):
        edge(e)
    edge(N - N % tile)                                  # the forward's last (partial) tile
    edge(N - N % 128)
    for r0, r1 in bwd_chunks(N, ws_chunk_rows):
        for e in range(r0, r1, REC_BAND_BLOCKS * 128):
            edge(e)
        for e in range(r0, r1, GRAD_BAND_ROWS):
            edge(e)
        edge(r1)
        edge(r1 - (r1 - r0) % 256)                      # last dH tile of the chunk
    rows.add(N - 1)
    return np.array(sorted(rows), dtype=np.int64)


def compare_forward(cfg, g, f, idx):
    """GPU per-row forward outputs at rows idx against the oracle's values f (same order)."""
    lse_err = float(np.abs(g["lse"][idx] - f["lse"]).max())
    logp_err = float(np.abs(g["logp"][idx] - f["logp"]).max())
    ratio_err = float((np.abs(g["ratio"][idx] - f["ratio"]) / f["ratio"]).max())
    near = np.minimum(np.abs(f["ratio"] - (1 + cfg.eps)), np.abs(f["ratio"] - (1 - cfg.eps))) < 1e-5
    cref = f["coef"][~near]
    coef_err = maxrel(g["coef"][idx][~near], cref) if cref.size else 0.0
    rl_err = maxrel(g["row_loss"][idx], f["row_loss"])
    stats = dict(rows=int(len(idx)), lse=lse_err, logp=logp_err, ratio=ratio_err, coef=coef_err, row_loss=rl_err,
                 near_clip=int(near.sum()))
    assert lse_err < 2e-4, stats
    assert logp_err < 2e-4, stats
    assert ratio_err < 2e-4, stats
    assert coef_err < 2e-4, stats
    assert rl_err < 2e-4, stats
    return stats


def check_head(cfg, b, g, pk, rows=None, grads=True, report=None):
    """Compare the head outputs with the oracle. rows: subset of packed rows (None = all)."""
    W = widen(cfg, b.W)
    idx = np.arange(len(pk["tok"])) if rows is None else np.asarray(rows, dtype=np.int64)
    Hs = widen(cfg, pk["hid"][idx])                    # only the rows the oracle evaluates
    f = lmhead.forward(Hs, W, pk["tok"][idx], pk["oldlogp"][idx], pk["adv"][idx], pk["w"][idx], cfg.eps,
                       cfg.loss_scale)
    stats = compare_forward(cfg, g, f, idx)
    if rows is None:
        rel = abs(g["loss"] - f["loss"]) / max(abs(f["loss"]), 1e-300)
        stats["loss_rel"] = rel
        assert rel < LOSS_RTOL, stats
    if grads:
        # the oracle's backward uses its own lse and coef
        if rows is None:
            dH, dW = lmhead.backward(Hs, W, pk["tok"], f["lse"], f["coef"])
            stats["dH"] = maxrel(g["dH"], dH)
            stats["dW"] = maxrel(g["dW"], dW)
        else:
            dH, _ = lmhead.backward(Hs, W, pk["tok"][idx], f["lse"], f["coef"], dw_vocab=[])
            stats["dH"] = maxrel(g["dH"][idx], dH)
        assert stats["dH"] < GRAD_MAXREL, stats
        if "dW" in stats:
            assert stats["dW"] < GRAD_MAXREL, stats
    if report is not None:
        report.update(stats)
        report["oracle_rows"], report["oracle_lse"], report["oracle_coef"] = idx, f["lse"], f["coef"]
    return stats
