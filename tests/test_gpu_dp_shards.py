"""The data-parallel split of the update pass on the product path, on one GPU.

A batch's prompts are split into contiguous shards, as data-parallel ranks would hold them
(whole groups, since advantages are per group). Each shard runs through libpsppo.so with the
global index of its first completion as traj_base (cutoffs are keyed by the global index), the
global loss scale 1/(P K) (Eq. full_update_G and Eq. truncated_update_Ghat: 1/K per prompt, the
mean over all P prompts), and PS_DW_ACCUMULATE on every shard after the first, so that dW sums
over the shards as an all-reduce would. Against the whole-batch pass: cutoffs, weights, packing
and every per-row output (lse, logp, ratio, coef, row loss, dH) bit for bit; the loss (a float64
sum) to 1e-12 relative; dW within the rounding of a different f32 accumulation order.

The dW bound: dW[v, c] sums the terms dZ_iv h_ic. The shards cut the rows into different 16-row
MMA steps and backward chunks (or, from the logit store, one launch over each pass's rows), so the
two results accumulate the same terms in another order.
Every accumulation step (a 16-deep MMA into the f32 accumulator in TMEM, or the addition of a
chunk's partial to dW) errs by at most 2 ulps (2^-22 relative) of a partial sum whose magnitude
is at most S[v, c] = sum_i |dZ_iv| |h_ic|. So |dW_shards - dW_whole| <= 2 n_acc 2^-22 S per entry,
with n_acc the longest chain of steps (rows per chunk / 16 plus the chunks), for either order.
"""
import numpy as np
import pytest
import torch

from synthetic import get_config, make_batch

from gpu_util import bwd_chunks

pytestmark = pytest.mark.gpu

def _abs_term_sums(hid, W, tok, lse, coef, rows=4096):
    """S[v, c] = sum_i |dZ_iv| |h_ic|, dZ = coef (onehot - softmax(z)): the magnitudes of the terms
    of dW[v, c] (plain torch f32; a bound, so its own rounding does not matter)."""
    S = torch.zeros(W.shape, dtype=torch.float32, device=W.device)
    Wf = W.float()
    for r0 in range(0, hid.shape[0], rows):
        h = hid[r0:r0 + rows].float()
        p = torch.exp(h @ Wf.T - lse[r0:r0 + rows, None])
        p[torch.arange(h.shape[0], device=h.device), tok[r0:r0 + rows].long()] -= 1.0
        S += p.abs_().mul_(coef[r0:r0 + rows, None].abs()).T @ h.abs()
    return S


ROW_OUTS = ("src_row", "row_traj", "row_pos", "tok", "oldlogp", "w", "adv", "lse", "logp", "ratio", "coef",
            "row_loss")


@pytest.mark.parametrize("name,world,store", [("mid", 2, False), ("1.5b", 2, False), ("1.5b", 3, False),
                                              ("mid", 2, True), ("1.5b", 3, True)])
def test_prompt_shards_reproduce_the_whole_batch(name, world, store):
    # store: the logits kept in the logit store by every pass (whole batch and shards); the shards'
    # backward converts each shard's store and accumulates dW over all of its rows in one launch
    from paper_2606_29758_gb300 import PS_MODE_TRUNC, PassShape, UpdatePass, prompt_shard
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    chunk = 65536 if cfg.V > 100000 else 256
    dt = torch.bfloat16
    whole = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, dt, chunk,
                                 b.total_len if store else 0), eps=cfg.eps,
                       loss_scale=cfg.loss_scale, mode=PS_MODE_TRUNC)
    N = whole.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    torch.cuda.synchronize()
    whole.check_status()

    dW = torch.full((cfg.V, cfg.d), float("nan"), dtype=torch.float32, device="cuda")
    loss = 0.0
    row0 = 0
    chunks = [r1 - r0 for r0, r1 in bwd_chunks(N, chunk)]
    for rank in range(world):
        sh = prompt_shard(cfg.P, cfg.K, b.L, world, rank)
        up = UpdatePass(PassShape(sh.prompts, cfg.K, b.T_max, cfg.d, cfg.V, sh.o1 - sh.o0, dt, chunk,
                                  sh.o1 - sh.o0 if store else 0), eps=cfg.eps,
                        loss_scale=cfg.loss_scale, mode=PS_MODE_TRUNC)     # the global scale 1/(P K)
        up.sample(D["q"][sh.p0:sh.p1], D["L"][sh.k0:sh.k1], cfg.seed, cfg.step, traj_base=sh.k0)
        n = up.pack(D["L"][sh.k0:sh.k1], D["R"][sh.k0:sh.k1], D["tok_full"][sh.o0:sh.o1],
                    D["oldlogp_full"][sh.o0:sh.o1], D["hid_full"][sh.o0:sh.o1])
        up.forward(D["W"])
        flags = B.PS_DW_ACCUMULATE if rank > 0 else B.PS_DW_OVERWRITE
        if store:
            assert up.stored and whole.stored is False      # the whole pass's backward has consumed its store
            B.ps_lmhead_ppo_bwd_from_store(n, cfg.d, cfg.V, up.dcode, up.hid, D["W"], up.tok, up.lse, up.logp,
                                           up.coef, up.store, up.dH, dW, flags, up.ws_bwd)
        else:
            B.ps_lmhead_ppo_bwd(n, cfg.d, cfg.V, up.dcode, up.hid, D["W"], up.tok, up.lse, up.coef, up.dH, dW,
                                flags, up.ws_bwd)
        torch.cuda.synchronize()
        up.check_status()
        # cutoffs, weights and packing: the whole batch's, shifted to the shard
        assert torch.equal(up.H, whole.H[sh.k0:sh.k1]) and torch.equal(up.n, whole.n[sh.k0:sh.k1])
        assert torch.equal(up.w_tab, whole.w_tab[sh.p0:sh.p1])
        cu = whole.cu_seqlens[sh.k0:sh.k1 + 1]
        assert torch.equal(up.cu_seqlens, cu - cu[0]) and int(cu[0]) == row0 and n == int(cu[-1] - cu[0])
        shift = {"src_row": sh.o0, "row_traj": sh.k0}
        for k in ROW_OUTS:
            got = getattr(up, k)[:n]
            ref = getattr(whole, k)[row0:row0 + n]
            assert torch.equal(got + shift.get(k, 0), ref), (rank, k)
        assert torch.equal(up.hid[:n], whole.hid[row0:row0 + n])
        assert torch.equal(up.dH[:n], whole.dH[row0:row0 + n]), rank
        loss += up.loss.item()
        row0 += n
        chunks = max(chunks, [r1 - r0 for r0, r1 in bwd_chunks(n, chunk)], key=lambda c: max(c) // 16 + len(c))
    assert row0 == N
    loss_rel = abs(loss - whole.loss.item()) / abs(whole.loss.item())
    diff = (dW - whole.dW).abs()
    # the store path's dW runs over all of a pass's rows in one launch, accumulated over the shards
    n_acc = -(-N // 16) + world if store else -(-max(chunks) // 16) + len(chunks)
    S = _abs_term_sums(whole.hid[:N], D["W"], whole.tok[:N], whole.lse[:N], whole.coef[:N])
    viol = (diff / (2 * n_acc * 2.0 ** -22 * S + 1e-30)).max().item()
    dw_rel = (diff.max() / whole.dW.abs().max()).item()
    fro = (diff.norm() / whole.dW.norm()).item()
    print(name, world, "store" if store else "recompute", "N", N, "loss rel", loss_rel, "dW max-rel", dw_rel, "Frobenius rel", fro,
          "worst entry / bound", viol, "n_acc", n_acc)
    assert loss_rel < 1e-12, loss_rel
    assert torch.isfinite(dW).all() and viol <= 1.0, viol
