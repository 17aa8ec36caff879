"""The oracle's LM-head forward (and dH rows) over many packed rows, on every host core.

Test infrastructure. The oracle's per-row quantities (Eq. 1 through the head of Appendix D: lse,
logp, ratio, row loss, coef, and the dH row of the backward) depend on that row alone, so a set
of rows splits into slices that worker processes evaluate with the unchanged oracle functions
(`oracle.lmhead.forward`, then `oracle.lmhead.backward` for the slice's dH rows with the slice's
own lse and coef). The parent concatenates the slices in row order; the loss over the rows is
`math.fsum` of the row losses, which is what `lmhead.forward` returns for the same rows in one call.

Workers are started with `spawn` (a pool forked from a process that has initialised CUDA can
hang) and run single-threaded BLAS, so the slices' exponentials run in parallel too. W is written
once, widened to float64, to a temporary file that every worker maps read-only.
"""
from __future__ import annotations

import math
import multiprocessing as mp
import os
import shutil
import tempfile

import numpy as np

SLICE_ROWS = 256


def _slice_task(args):
    cfg, w_path, w_shape, hid, tok, oldlogp, adv, w, want_dh = args
    from oracle import lmhead
    from oracle.pipeline import widen
    W = np.memmap(w_path, dtype=np.float64, mode="r", shape=w_shape)
    H = widen(cfg, hid)
    f = lmhead.forward(H, W, tok, oldlogp, adv, w, cfg.eps, cfg.loss_scale)
    out = {k: f[k] for k in ("lse", "logp", "ratio", "row_loss", "coef")}
    if want_dh.any():
        dh_rows = np.nonzero(want_dh)[0]
        out["dH"], _ = lmhead.backward(H, W, tok, f["lse"], f["coef"], dh_rows=dh_rows, dw_vocab=[])
        out["dh_rows"] = dh_rows
    return out


def oracle_rows(cfg, W_bits, hid_rows, tok, oldlogp, adv, w, dh_mask=None, workers=None):
    """Oracle forward over the given packed rows (hid_rows: bf16 bits or f32, in row order), and
    the dH row wherever dh_mask is set. Returns per-row float64 arrays, `dH` [sum(dh_mask), d] in row
    order, and `loss` = fsum of the row losses."""
    from oracle.pipeline import widen
    n = len(tok)
    dh_mask = np.zeros(n, dtype=bool) if dh_mask is None else np.asarray(dh_mask, dtype=bool)
    workers = workers or min(os.cpu_count() or 1, 16)
    tmp = tempfile.mkdtemp(prefix="oracle_w_")
    try:
        w_path = os.path.join(tmp, "W.f64")
        W64 = np.memmap(w_path, dtype=np.float64, mode="w+", shape=W_bits.shape)
        for r0 in range(0, W_bits.shape[0], 8192):
            W64[r0:r0 + 8192] = widen(cfg, W_bits[r0:r0 + 8192])
        W64.flush()
        del W64
        tasks = [(cfg, w_path, W_bits.shape, hid_rows[s:s + SLICE_ROWS], tok[s:s + SLICE_ROWS],
                  oldlogp[s:s + SLICE_ROWS], adv[s:s + SLICE_ROWS], w[s:s + SLICE_ROWS], dh_mask[s:s + SLICE_ROWS])
                 for s in range(0, n, SLICE_ROWS)]
        saved = {k: os.environ.get(k) for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS")}
        for k in saved:
            os.environ[k] = "1"
        try:
            with mp.get_context("spawn").Pool(workers) as pool:
                parts = pool.map(_slice_task, tasks, chunksize=1)
        finally:
            for k, v in saved.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v
    finally:
        shutil.rmtree(tmp, ignore_errors=True)
    res = {k: np.concatenate([p[k] for p in parts]) for k in ("lse", "logp", "ratio", "row_loss", "coef")}
    dh = [p["dH"] for p in parts if "dH" in p]
    res["dH"] = np.concatenate(dh) if dh else np.zeros((0, W_bits.shape[1]))
    res["loss"] = math.fsum(res["row_loss"].tolist())
    return res
