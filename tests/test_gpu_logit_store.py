"""The logit store: the forward keeps its logits and the backward turns them into dZ in place.

Against the recompute path on the same batch and against the oracle (Eq. 1 through the head of
Appendix D):
- the forward's outputs (lse, logp, ratio, coef, row loss, loss) are bit-identical to the recompute
  path's: the store epilogue sums the same e_v = 2^(x_v - m) in the same order;
- after the forward the store holds, for every row and column, e = 2^(x - m) in f16 with x = z log2 e
  and m the scale of the column's 32-column slice: against the oracle's logits, within the f16
  rounding of e (2^-11 relative at or above 2^-14, 2^-24 absolute below) and the f32 accumulation of
  z (1e-4 relative, generous), and e <= 1;
- after the backward it holds dZ in bf16: against coef (1[v = o] - exp(z - lse)) evaluated from the
  oracle's logits with the pass's own lse and coef, per element within the bf16 rounding of dZ (unit
  roundoff 2^-8), the f16 rounding of e (2^-11 relative) and the accumulation of z
  (2^-22 |coef| + 1e-4 |coef| p);
- dH and dW match the oracle within the path's 2e-2 max-relative tolerance.
Ragged shapes (a 9-column last slice, a vocabulary that is not a multiple of 8 in the row pitch,
rows that end inside a 32-row conversion block and a 128-row tile), tokens on slice and pitch edges,
the accumulate flags and N = 0 are covered on a hand-built head.
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

from oracle import lmhead
from oracle.pipeline import widen
from synthetic import get_config, make_batch

from gpu_util import GRAD_MAXREL, maxrel, oracle_prefix, schedule_rows
from oracle_pool import oracle_rows

pytestmark = pytest.mark.gpu

LOG2E = 1.4426950408889634
OUTS = ("lse", "logp", "ratio", "coef", "row_loss")


def _store_views(store, N, V):
    """(e f16 [N][V], m f32 [ceil(V/32)][N], dZ bf16 [N][V]) views of a store of N rows."""
    ldz = -(-V // 8) * 8
    nz = N * ldz * 2
    off = -(-nz // 256) * 256
    nc = -(-V // 32)
    e = store[:nz].view(torch.float16).view(N, ldz)[:, :V]
    m = store[off:off + 4 * nc * N].view(torch.float32).view(nc, N)
    dz = store[:nz].view(torch.bfloat16).view(N, ldz)[:, :V]
    return e, m, dz


def _check_e(e, m, z):
    """e [n][V] (float64 of the stored f16), m [n][nc] the rows' slice scales, z [n][V] oracle logits."""
    V = z.shape[1]
    e_ref = np.exp2(z * LOG2E - m[:, np.arange(V) // 32])
    assert np.all(e <= 1.0) and np.all(e >= 0.0)
    tol = np.where(e_ref >= 2.0 ** -14, (2.0 ** -11 + 1e-4) * e_ref, 2.0 ** -24 + 1e-4 * e_ref)
    bad = np.abs(e - e_ref) > tol
    assert not bad.any(), (int(bad.sum()), float((np.abs(e - e_ref) / tol).max()))


def _check_dz(dz, z, tok, lse, coef):
    """dz [n][V] (float64 of the stored bf16) against coef (onehot - exp(z - lse)) with the pass's lse, coef."""
    p = np.exp(z - lse[:, None])
    ref = -coef[:, None] * p
    r = np.arange(len(tok))
    ref[r, tok] += coef
    tol = (2.0 ** -8 + 2.0 ** -11) * np.abs(ref) + np.abs(coef)[:, None] * (2.0 ** -22 + 1e-4 * p)
    diff = np.abs(dz - ref)
    # rows with coef = 0 (clip bound, zero advantage) must be exactly zero
    ratio = np.where(tol > 0, diff / np.where(tol > 0, tol, 1.0), np.where(diff > 0, np.inf, 0.0))
    assert ratio.max() <= 1.0, (float(ratio.max()), np.unravel_index(ratio.argmax(), ratio.shape))
    return float(ratio.max())


def _two_passes(cfg, b, store_rows=None):
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    shape = PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, 65536)
    rec = UpdatePass(shape, eps=cfg.eps, loss_scale=cfg.loss_scale)
    sto = UpdatePass(replace(shape, store_rows=b.total_len if store_rows is None else store_rows), eps=cfg.eps,
                     loss_scale=cfg.loss_scale)
    return rec, sto


@pytest.mark.parametrize("name", ["mid", "head7b_small", "head1.5b_small"])
def test_store_matches_the_recompute_path_and_the_oracle(name):
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    rec, sto = _two_passes(cfg, b)
    args = (D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    N = rec.run(*args)
    sto.sample(D["q"], D["L"], cfg.seed, cfg.step)
    assert sto.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"]) == N
    sto.forward(D["W"])
    torch.cuda.synchronize()
    assert sto.stored
    for k in OUTS:
        assert torch.equal(getattr(sto, k)[:N], getattr(rec, k)[:N]), k
    assert sto.loss.item() == rec.loss.item()

    _, _, _, _, pk = oracle_prefix(cfg, b)
    Hs, W64 = widen(cfg, pk["hid"]), widen(cfg, b.W)
    e, m, _ = _store_views(sto.store, N, cfg.V)
    m_np = m.cpu().numpy().astype(np.float64).T                 # [N][nc]
    e_np = e.float().cpu().numpy().astype(np.float64)
    for r0 in range(0, N, 64):
        z = lmhead.logits(Hs[r0:r0 + 64], W64)
        _check_e(e_np[r0:r0 + 64], m_np[r0:r0 + 64], z)

    sto.backward(D["W"])
    torch.cuda.synchronize()
    sto.check_status()
    rec.check_status()
    _, _, dz = _store_views(sto.store, N, cfg.V)
    dz_np = dz.float().cpu().numpy().astype(np.float64)
    lse = sto.lse[:N].double().cpu().numpy()
    coef = sto.coef[:N].double().cpu().numpy()
    worst = 0.0
    for r0 in range(0, N, 64):
        z = lmhead.logits(Hs[r0:r0 + 64], W64)
        worst = max(worst, _check_dz(dz_np[r0:r0 + 64], z, pk["tok"][r0:r0 + 64], lse[r0:r0 + 64],
                                     coef[r0:r0 + 64]))
    f = lmhead.forward(Hs, W64, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], cfg.eps, cfg.loss_scale)
    dH_ref, dW_ref = lmhead.backward(Hs, W64, pk["tok"], f["lse"], f["coef"])
    e_h = maxrel(sto.dH[:N].double().cpu().numpy(), dH_ref)
    e_w = maxrel(sto.dW.double().cpu().numpy(), dW_ref)
    e_rh = maxrel(rec.dH[:N].double().cpu().numpy(), dH_ref)
    e_rw = maxrel(rec.dW.double().cpu().numpy(), dW_ref)
    print(name, N, "dZ worst / bound", worst, "dH", e_h, "dW", e_w, "(recompute path: dH", e_rh, "dW", e_rw, ")")
    assert e_h < GRAD_MAXREL and e_w < GRAD_MAXREL


def _ragged_head(N, d=64, V=1001, seed=7):
    rng = np.random.default_rng(seed)
    H = rng.standard_normal((N, d)).astype(np.float32)
    W = (rng.standard_normal((V, d)) * 0.3).astype(np.float32)
    tok = rng.integers(0, V, N).astype(np.int32)
    edges = [0, 31, 32, 991, 992, 999, 1000, 1000, 500, 7]
    tok[:len(edges)] = edges
    # a peaked row: its chosen logit near 14, p(o) about 0.997
    H[9] = 14.0 * W[tok[9]] / float(W[tok[9]] @ W[tok[9]])
    oldlogp = (rng.standard_normal(N) * 0.3 - 3.0).astype(np.float32)
    oldlogp[9] = -0.01
    adv = rng.standard_normal(N).astype(np.float32)
    w = rng.uniform(1.0, 3.0, N).astype(np.float32)
    Hb = torch.from_numpy(H).to(torch.bfloat16)
    Wb = torch.from_numpy(W).to(torch.bfloat16)
    return Hb, Wb, tok, oldlogp, adv, w


@pytest.mark.parametrize("N", [37, 300])
def test_store_on_ragged_shapes_with_accumulation(N):
    from paper_2606_29758_gb300 import _binding as B
    d, V = 64, 1001
    Hb, Wb, tok, oldlogp, adv, w = _ragged_head(N, d, V)
    dev = dict(device="cuda")
    Hd, Wd = Hb.cuda(), Wb.cuda()
    tk, ol, ad, ww = (torch.from_numpy(a).cuda() for a in (tok, oldlogp, adv, w))
    outs = {k: torch.empty(N, dtype=torch.float32, **dev) for k in OUTS}
    loss = torch.zeros(1, dtype=torch.float64, **dev)
    ws_f = torch.zeros(B.ps_lmhead_ppo_fwd_workspace_size(N, d, V, B.PS_DTYPE_BF16), dtype=torch.uint8, **dev)
    ws_b = torch.zeros(B.ps_lmhead_ppo_bwd_from_store_workspace_size(), dtype=torch.uint8, **dev)
    store = torch.empty(B.ps_lmhead_logit_store_size(N, V) + 4096, dtype=torch.uint8, **dev)   # larger is fine
    eps, scale = 0.2, 0.05

    def fwd():
        B.ps_lmhead_ppo_fwd_store(N, d, V, B.PS_DTYPE_BF16, Hd, Wd, tk, ol, ad, ww, eps, scale, loss, outs["lse"],
                                  outs["logp"], outs["ratio"], outs["coef"], outs["row_loss"], store, ws_f)

    fwd()
    torch.cuda.synchronize()
    e, m, _ = _store_views(store, N, V)
    H64, W64 = Hb.double().numpy(), Wb.double().numpy()
    z = lmhead.logits(H64, W64)
    _check_e(e.float().cpu().numpy().astype(np.float64), m.cpu().numpy().astype(np.float64).T, z)
    f = lmhead.forward(H64, W64, tok, oldlogp.astype(np.float64), adv.astype(np.float64), w.astype(np.float64),
                       eps, scale)
    assert abs(loss.item() - f["loss"]) <= 1e-5 * abs(f["loss"])
    np.testing.assert_allclose(outs["lse"].cpu().numpy(), f["lse"], rtol=0, atol=2e-5)
    assert f["logp"][9] > np.log(0.98)                          # the peaked row is peaked

    dH = torch.full((N, d), float("nan"), **dev)
    dW = torch.full((V, d), float("nan"), **dev)
    B.ps_lmhead_ppo_bwd_from_store(N, d, V, B.PS_DTYPE_BF16, Hd, Wd, tk, outs["lse"], outs["logp"], outs["coef"],
                                   store, dH, dW, B.PS_DW_OVERWRITE, ws_b)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws_f)[0] == B.PS_OK and B.ps_workspace_status(ws_b)[0] == B.PS_OK
    _, _, dz = _store_views(store, N, V)
    _check_dz(dz.float().cpu().numpy().astype(np.float64), z, tok, outs["lse"].double().cpu().numpy(),
              outs["coef"].double().cpu().numpy())
    dH_ref, dW_ref = lmhead.backward(H64, W64, tok, f["lse"], f["coef"])
    assert maxrel(dH.double().cpu().numpy(), dH_ref) < GRAD_MAXREL
    assert maxrel(dW.double().cpu().numpy(), dW_ref) < GRAD_MAXREL

    # the accumulate flags add the same products to what the buffers hold (the kernels are deterministic)
    fwd()
    pre_h = torch.randn(N, d, **dev)
    pre_w = torch.randn(V, d, **dev)
    dH2, dW2 = pre_h.clone(), pre_w.clone()
    B.ps_lmhead_ppo_bwd_from_store(N, d, V, B.PS_DTYPE_BF16, Hd, Wd, tk, outs["lse"], outs["logp"], outs["coef"],
                                   store, dH2, dW2, B.PS_DW_ACCUMULATE | B.PS_DH_ACCUMULATE, ws_b)
    torch.cuda.synchronize()
    assert torch.equal(dH2, pre_h + dH) and torch.equal(dW2, pre_w + dW)


def test_store_with_no_rows():
    from paper_2606_29758_gb300 import _binding as B
    d, V = 64, 1001
    dev = dict(device="cuda")
    e1 = torch.empty(1, dtype=torch.float32, **dev)
    i1 = torch.empty(1, dtype=torch.int32, **dev)
    h1 = torch.empty(1, d, dtype=torch.bfloat16, **dev)
    Wd = torch.randn(V, d, **dev).to(torch.bfloat16)
    loss = torch.full((1,), 7.0, dtype=torch.float64, **dev)
    store = torch.empty(16, dtype=torch.uint8, **dev)
    ws_f = torch.zeros(B.ps_lmhead_ppo_fwd_workspace_size(0, d, V, B.PS_DTYPE_BF16), dtype=torch.uint8, **dev)
    B.ps_lmhead_ppo_fwd_store(0, d, V, B.PS_DTYPE_BF16, h1, Wd, i1, e1, e1, e1, 0.2, 1.0, loss, e1, e1, e1, e1, None,
                              store, ws_f)
    dW = torch.full((V, d), 3.0, **dev)
    ws_b = torch.zeros(B.ps_lmhead_ppo_bwd_from_store_workspace_size(), dtype=torch.uint8, **dev)
    B.ps_lmhead_ppo_bwd_from_store(0, d, V, B.PS_DTYPE_BF16, h1, Wd, i1, e1, e1, e1, store, None, dW,
                                   B.PS_DW_OVERWRITE, ws_b)
    torch.cuda.synchronize()
    assert loss.item() == 0.0 and float(dW.abs().max()) == 0.0


@pytest.mark.parametrize("name", ["7b", "1.5b"])
def test_store_at_full_size(name):
    # a full-size workload through the store path: the forward bit-identical to the recompute path's; dH on a stratified set of rows (every 128-row block, the forward's band edges,
    # the dH bands and the last tile) and dZ on about 96 of them against the oracle; sum_v dW = 0; dW
    # against the recompute path's
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    rec, sto = _two_passes(cfg, b)
    args = (D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    N = rec.run(*args)
    sto.sample(D["q"], D["L"], cfg.seed, cfg.step)
    assert sto.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"]) == N
    sto.forward(D["W"])
    torch.cuda.synchronize()
    for k in OUTS:
        assert torch.equal(getattr(sto, k)[:N], getattr(rec, k)[:N]), k
    assert sto.loss.item() == rec.loss.item()
    sto.backward(D["W"])
    torch.cuda.synchronize()
    sto.check_status()
    rec.check_status()

    _, _, _, _, pk = oracle_prefix(cfg, b)
    rows = schedule_rows(cfg, N, N)                             # one chunk: the store's dH runs over all rows
    res = oracle_rows(cfg, b.W, pk["hid"][rows], pk["tok"][rows], pk["oldlogp"][rows], pk["adv"][rows],
                      pk["w"][rows], dh_mask=np.ones(len(rows), dtype=bool))
    g_dH = sto.dH[torch.from_numpy(rows).cuda()].double().cpu().numpy()
    err_h = maxrel(g_dH, res["dH"])
    assert err_h < GRAD_MAXREL, err_h

    rng = np.random.default_rng(5)
    sub = np.unique(np.concatenate([rows[:8], rows[-8:], rng.choice(rows, 80, replace=False)]))
    _, _, dz = _store_views(sto.store, N, cfg.V)
    sel = torch.from_numpy(sub).cuda()
    dz_np = dz[sel].float().cpu().numpy().astype(np.float64)
    W64 = widen(cfg, b.W)
    z = lmhead.logits(widen(cfg, pk["hid"][sub]), W64)
    worst = _check_dz(dz_np, z, pk["tok"][sub], sto.lse[sel].double().cpu().numpy(),
                      sto.coef[sel].double().cpu().numpy())

    colsum = sto.dW.double().sum(dim=0)
    bound = (sto.coef[:N].abs()[:, None] * sto.hid[:N].float().abs()).double().sum(dim=0) * 2.0 ** -8
    assert (colsum.abs() / (1.5 * bound + 1e-6 * sto.dW.abs().max().double())).max().item() < 1.0
    err_w = (sto.dW - rec.dW).abs().max().item() / rec.dW.abs().max().item()
    print(name, N, "rows", len(rows), "dH max-rel", err_h, "dZ worst / bound", worst, "dW store vs recompute", err_w)
    assert err_w < 1e-2
    assert torch.isfinite(sto.dW).all() and torch.isfinite(sto.dH[:N]).all()


def test_update_pass_recomputes_when_the_store_is_too_small():
    # a step with more rows than the store holds takes the recompute path (bit-identical to a pass
    # without a store); one that fits takes the store
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    D = b.dev
    rec, _ = _two_passes(cfg, b, store_rows=0)
    args = (D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    N = rec.run(*args)
    _, small = _two_passes(cfg, b, store_rows=N - 1)
    _, fits = _two_passes(cfg, b, store_rows=N)
    assert small.run(*args, grads=False) == N and not small.stored
    assert fits.run(*args, grads=False) == N and fits.stored
    small.backward(D["W"])
    fits.backward(D["W"])
    torch.cuda.synchronize()
    for up in (rec, small, fits):
        up.check_status()
    assert torch.equal(small.dH[:N], rec.dH[:N]) and torch.equal(small.dW, rec.dW)
    assert small.loss.item() == rec.loss.item() == fits.loss.item()
    assert not torch.equal(fits.dW, rec.dW)          # the store's dZ rounds differently
    assert maxrel(fits.dW.double().cpu().numpy(), rec.dW.double().cpu().numpy()) < 1e-2
