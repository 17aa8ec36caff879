"""The vocabulary-parallel head, its shards run one after another on one GPU.

W is split by vocabulary rows into S shards. Each shard's per-row logit statistics (base-2 maximum,
sum of powers, the chosen logit where the token falls in the shard) are combined into the forward's
outputs, and each shard's backward gives its rows of dW and its term of dH (PS_DH_ACCUMULATE sums
the terms here, as an all-reduce would across devices). Against the whole-head pass of the library
(Eq. 1 through the head of Appendix D), and against the oracle:
- with the whole head's lse and coef, every shard's dW rows are bit-identical to the whole head's
  (the same recomputed logits, accumulated over the same rows in the same chunks and order), and the
  summed dH agrees within the rounding of a different accumulation order: dH[i, c] sums the terms
  dZ_iv W_vc over the vocabulary, one accumulator in the whole head, S partial sums added to one
  another here; every accumulation step (a 16-deep MMA, or the addition of a shard's term) errs by
  at most 2 ulps (2^-22 relative) of a partial sum, whose magnitude is at most
  T[i, c] = sum_v |dZ_iv| |W_vc|, so |dH_shards - dH_whole| <= 2 n_acc 2^-22 T per entry, with n_acc =
  ceil(V / 16) + S the longest chain of steps (a missing or doubled shard term breaks it by far);
- the forward from the shards' statistics agrees with the whole head's to rounding (the per-row
  sums merge in another grouping), and its lse, coef and the resulting gradients match the oracle
  within the path's tolerances.
"""
import numpy as np
import pytest
import torch

from synthetic import get_config, make_batch

from gpu_util import GRAD_MAXREL, LOSS_RTOL, compare_forward, maxrel, oracle_prefix

pytestmark = pytest.mark.gpu

OUTS = ("lse", "logp", "ratio", "coef", "row_loss")


def _dh_term_sums(hid, W, tok, lse, coef, rows=2048):
    """T[i, c] = sum_v |dZ_iv| |W_vc|, dZ = coef (onehot - softmax(z)): the magnitudes of the terms
    of dH[i, c] (plain torch f32; a bound, so its own rounding does not matter)."""
    Wf = W.float()
    Wa = Wf.abs()
    T = torch.empty(hid.shape[0], W.shape[1], dtype=torch.float32, device=W.device)
    for r0 in range(0, hid.shape[0], rows):
        h = hid[r0:r0 + rows].float()
        p = torch.exp(h @ Wf.T - lse[r0:r0 + rows, None])
        p[torch.arange(h.shape[0], device=h.device), tok[r0:r0 + rows].long()] -= 1.0
        T[r0:r0 + rows] = p.abs_().mul_(coef[r0:r0 + rows, None].abs()) @ Wa
    return T


def _check_dh(tag, dH, ref, hid, W, tok, lse, coef, V, S):
    n_acc = -(-V // 16) + S
    bound = 2 * n_acc * 2.0 ** -22 * _dh_term_sums(hid, W, tok, lse, coef)
    diff = (dH - ref).abs()
    viol = (diff / (bound + 1e-30)).max().item()
    print(tag, "dH max-rel vs the whole head", (diff.max() / ref.abs().max()).item(), "worst entry / bound", viol)
    assert torch.isfinite(dH).all() and viol <= 1.0, viol


def _shard_layouts(V):
    from paper_2606_29758_gb300 import vocab_shards
    return [vocab_shards(V, 3), [(0, 5), (5, V - 305), (V - 300, 300)]]


@pytest.mark.parametrize("name", ["mid", "mid_f32", "head7b_small"])
def test_vocab_shards_reproduce_the_whole_head(name):
    from paper_2606_29758_gb300 import PassShape, UpdatePass, VocabParallelHead
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, dt, 256), eps=cfg.eps,
                    loss_scale=cfg.loss_scale)
    N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    torch.cuda.synchronize()
    up.check_status()
    _, _, _, _, pk = oracle_prefix(cfg, b)
    W = D["W"]
    for shards in _shard_layouts(cfg.V):
        vp = VocabParallelHead(shards, b.total_len, cfg.d, cfg.V, dt, eps=cfg.eps, loss_scale=cfg.loss_scale,
                               bwd_chunk_rows=256)
        for r, (v0, Vs) in enumerate(shards):
            vp.stats(r, N, up.hid, W[v0:v0 + Vs], up.tok)
        vp.forward(N, up.tok, up.oldlogp, up.adv, up.w)
        torch.cuda.synchronize()
        for k in OUTS:
            ref, got = getattr(up, k)[:N], getattr(vp, k)[:N]
            tol = 2e-5 * max(1.0, ref.abs().max().item())
            assert (got - ref).abs().max().item() <= tol, (k, shards)
        assert abs(vp.loss.item() - up.loss.item()) <= 1e-5 * abs(up.loss.item())

        # backward with the whole head's lse and coef: the shards' dW rows are the whole head's, bit for bit
        vp.lse.copy_(up.lse)
        vp.coef.copy_(up.coef)
        dH = torch.full_like(up.dH, float("nan"))
        dW = torch.full_like(up.dW, float("nan"))
        for r, (v0, Vs) in enumerate(shards):
            vp.backward(r, N, up.hid, W[v0:v0 + Vs], up.tok, dH, dW[v0:v0 + Vs], add_to_dH=r > 0)
        torch.cuda.synchronize()
        for ws in (vp.ws_stats, vp.ws_fin, vp.ws_bwd):
            assert B.ps_workspace_status(ws)[0] == B.PS_OK
        assert torch.equal(dW, up.dW), (dW - up.dW).abs().max().item()
        _check_dh(f"{name} {shards}", dH[:N], up.dH[:N], up.hid[:N], W, up.tok[:N], up.lse[:N], up.coef[:N],
                  cfg.V, len(shards))

    # the sharded forward and backward against the oracle (every row)
    vp.forward(N, up.tok, up.oldlogp, up.adv, up.w)
    for r, (v0, Vs) in enumerate(shards):
        vp.backward(r, N, up.hid, W[v0:v0 + Vs], up.tok, dH, dW[v0:v0 + Vs], add_to_dH=r > 0)
    torch.cuda.synchronize()
    from oracle import lmhead
    from oracle.pipeline import widen
    Hs, W64 = widen(cfg, pk["hid"]), widen(cfg, b.W)
    f = lmhead.forward(Hs, W64, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], cfg.eps, cfg.loss_scale)
    g = {k: getattr(vp, k)[:N].cpu().numpy() for k in OUTS}
    compare_forward(cfg, g, f, np.arange(N))
    assert abs(vp.loss.item() - f["loss"]) / abs(f["loss"]) < LOSS_RTOL
    dH_ref, dW_ref = lmhead.backward(Hs, W64, pk["tok"], f["lse"], f["coef"])
    assert maxrel(dH[:N].double().cpu().numpy(), dH_ref) < GRAD_MAXREL
    assert maxrel(dW.double().cpu().numpy(), dW_ref) < GRAD_MAXREL


def test_vocab_shards_at_the_7b_head_with_several_chunks():
    # the 7B-shaped head on ~25k packed rows: several backward chunks and row bands per shard
    from paper_2606_29758_gb300 import PassShape, UpdatePass, VocabParallelHead, vocab_shards
    cfg = get_config("7b_p2")
    b = make_batch(cfg, device="cuda")
    D = b.dev
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, 8192),
                    eps=cfg.eps, loss_scale=cfg.loss_scale)
    N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    shards = vocab_shards(cfg.V, 4)
    vp = VocabParallelHead(shards, b.total_len, cfg.d, cfg.V, torch.bfloat16, eps=cfg.eps,
                           loss_scale=cfg.loss_scale, bwd_chunk_rows=8192)
    W = D["W"]
    for r, (v0, Vs) in enumerate(shards):
        vp.stats(r, N, up.hid, W[v0:v0 + Vs], up.tok)
    vp.forward(N, up.tok, up.oldlogp, up.adv, up.w)
    torch.cuda.synchronize()
    up.check_status()
    for k in OUTS:
        ref, got = getattr(up, k)[:N], getattr(vp, k)[:N]
        assert (got - ref).abs().max().item() <= 2e-5 * max(1.0, ref.abs().max().item()), k
    assert abs(vp.loss.item() - up.loss.item()) <= 1e-5 * abs(up.loss.item())
    vp.lse.copy_(up.lse)
    vp.coef.copy_(up.coef)
    dH = torch.empty_like(up.dH)
    dW = torch.empty_like(up.dW)
    for r, (v0, Vs) in enumerate(shards):
        vp.backward(r, N, up.hid, W[v0:v0 + Vs], up.tok, dH, dW[v0:v0 + Vs], add_to_dH=r > 0)
    torch.cuda.synchronize()
    assert torch.equal(dW, up.dW)
    _check_dh(f"7b_p2 {N}", dH[:N], up.dH[:N], up.hid[:N], W, up.tok[:N], up.lse[:N], up.coef[:N], cfg.V,
              len(shards))


@pytest.mark.parametrize("name", ["mid", "head7b_small"])
def test_vocab_shards_with_logit_stores(name):
    # every shard keeps its logits in a store of its own (ps_lmhead_logit_stats_store) and its backward
    # converts it (ps_lmhead_ppo_bwd_vocab_shard_from_store): the statistics equal the plain calls' bit for
    # bit (the same sums in the same order), and the gradients match the oracle and the shards that
    # recompute
    from paper_2606_29758_gb300 import PassShape, UpdatePass, VocabParallelHead
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, 256), eps=cfg.eps,
                    loss_scale=cfg.loss_scale)
    N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    torch.cuda.synchronize()
    _, _, _, _, pk = oracle_prefix(cfg, b)
    W = D["W"]
    from oracle import lmhead
    from oracle.pipeline import widen
    Hs, W64 = widen(cfg, pk["hid"]), widen(cfg, b.W)
    f = lmhead.forward(Hs, W64, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"], cfg.eps, cfg.loss_scale)
    dH_ref, dW_ref = lmhead.backward(Hs, W64, pk["tok"], f["lse"], f["coef"])
    for shards in _shard_layouts(cfg.V):
        heads = {}
        for store in (False, True):
            vp = VocabParallelHead(shards, b.total_len, cfg.d, cfg.V, torch.bfloat16, eps=cfg.eps,
                                   loss_scale=cfg.loss_scale, bwd_chunk_rows=256, store=store)
            for r, (v0, Vs) in enumerate(shards):
                vp.stats(r, N, up.hid, W[v0:v0 + Vs], up.tok)
            vp.forward(N, up.tok, up.oldlogp, up.adv, up.w)
            dH = torch.full_like(up.dH, float("nan"))
            dW = torch.full_like(up.dW, float("nan"))
            for r, (v0, Vs) in enumerate(shards):
                vp.backward(r, N, up.hid, W[v0:v0 + Vs], up.tok, dH, dW[v0:v0 + Vs], add_to_dH=r > 0)
            torch.cuda.synchronize()
            heads[store] = (vp, dH, dW)
        plain, stored = heads[False][0], heads[True][0]
        assert torch.equal(stored.stats_all[:, :N], plain.stats_all[:, :N])
        assert torch.equal(stored.ztok_all[:, :N], plain.ztok_all[:, :N])
        assert stored.loss.item() == plain.loss.item()
        _, dH_s, dW_s = heads[True]
        _, dH_p, dW_p = heads[False]
        e_h = maxrel(dH_s[:N].double().cpu().numpy(), dH_ref)
        e_w = maxrel(dW_s.double().cpu().numpy(), dW_ref)
        print(name, shards, "store: dH", e_h, "dW", e_w, "vs recomputing shards: dW",
              maxrel(dW_s.double().cpu().numpy(), dW_p.double().cpu().numpy()))
        assert torch.isfinite(dH_s[:N]).all() and torch.isfinite(dW_s).all()
        assert e_h < GRAD_MAXREL and e_w < GRAD_MAXREL
