"""The allocation-free forward (ps_lmhead_ppo_fwd_noalloc) against the workspace forward.

Callers that cannot allocate device memory (a plugin inside a framework that owns the GPU's
memory pool, a deployment with a fixed device memory plan) use the variant whose scratch is a
static device array inside the library. It must give the same outputs as ps_lmhead_ppo_fwd,
call after call (the array keeps the previous call's contents). This file is collected last.
"""
import pytest
import torch

from synthetic import get_config, make_batch

pytestmark = pytest.mark.gpu

OUTS = ("lse", "logp", "ratio", "coef", "row_loss")


def _prepared(name):
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, dt), eps=cfg.eps,
                    loss_scale=cfg.loss_scale)
    D = b.dev
    up.sample(D["q"], D["L"], cfg.seed, cfg.step)
    up.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"])
    up.forward(D["W"])              # the existing entry point, with a caller workspace
    torch.cuda.synchronize()
    up.check_status()
    return cfg, D, up


@pytest.mark.parametrize("name", ["mid", "head7b_small", "tiny"])
def test_noalloc_forward_matches_workspace_forward_twice(name):
    from paper_2606_29758_gb300 import _binding as B
    cfg, D, up = _prepared(name)
    N = up.N
    for call in range(2):
        out = {k: torch.full((N,), float("nan"), device="cuda") for k in OUTS}
        loss = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
        B.ps_lmhead_ppo_fwd_noalloc(N, cfg.d, cfg.V, up.dcode, up.hid, D["W"], up.tok, up.oldlogp, up.adv, up.w,
                                    cfg.eps, cfg.loss_scale, loss, out["lse"], out["logp"], out["ratio"],
                                    out["coef"], out["row_loss"])
        torch.cuda.synchronize()
        rel = abs(loss.item() - up.loss.item()) / abs(up.loss.item())
        assert rel < 1e-3, (call, rel)
        for k in OUTS:
            ref = getattr(up, k)[:N]
            err = (out[k] - ref).abs().max().item()
            assert err <= 2e-4 * max(1.0, ref.abs().max().item()), (call, k, err)


def test_noalloc_rejects_problems_larger_than_its_scratch():
    # 6 million rows need more than 64 MiB even with one vocabulary range per row: refused before any launch
    # (the pointers are valid but never read).
    from paper_2606_29758_gb300 import _binding as B
    t = torch.zeros(64, device="cuda")
    with pytest.raises(B.PsppoError) as e:
        B.ps_lmhead_ppo_fwd_noalloc(6_000_000, 3584, 152064, B.PS_DTYPE_BF16, t, t, t, t, t, t,
                                    0.2, 1.0, t, t, t, t, t, t)
    assert e.value.status == B.PS_ERR_UNSUPPORTED


def test_noalloc_bad_token_shows_as_nan_in_its_row_and_the_loss():
    # No workspace comes back from this call, so its status word cannot be read: a token id
    # outside [0, V) must show as NaN in that row's outputs and in the loss, and nowhere else.
    from paper_2606_29758_gb300 import _binding as B
    cfg, D, up = _prepared("mid")
    N = up.N
    bad = N // 3
    tok = up.tok[:N].clone()
    tok[bad] = cfg.V
    out = {k: torch.zeros(N, device="cuda") for k in OUTS}
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    B.ps_lmhead_ppo_fwd_noalloc(N, cfg.d, cfg.V, up.dcode, up.hid, D["W"], tok, up.oldlogp, up.adv, up.w,
                                cfg.eps, cfg.loss_scale, loss, out["lse"], out["logp"], out["ratio"],
                                out["coef"], out["row_loss"])
    torch.cuda.synchronize()
    assert torch.isnan(loss).all()
    for k in ("logp", "ratio", "row_loss"):
        assert torch.isnan(out[k][bad]), k
    keep = torch.ones(N, dtype=torch.bool, device="cuda")
    keep[bad] = False
    for k in OUTS:
        assert torch.isfinite(out[k][keep]).all(), k
        assert torch.equal(out[k][keep], getattr(up, k)[:N][keep]), k   # every other row as before


def test_noalloc_with_fewer_vocabulary_partials_than_tiles():
    # About 25k packed rows of the 7B-shaped head (V = 152064): the static scratch holds fewer than
    # the ceil(V / 256) partials per row, so the forward runs with contiguous vocabulary ranges.
    from paper_2606_29758_gb300 import _binding as B
    cfg, D, up = _prepared("7b_p2")
    N = up.N
    assert N * 8 * ((cfg.V + 255) // 256) > (64 << 20)
    for call in range(2):
        out = {k: torch.full((N,), float("nan"), device="cuda") for k in OUTS}
        loss = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
        B.ps_lmhead_ppo_fwd_noalloc(N, cfg.d, cfg.V, up.dcode, up.hid, D["W"], up.tok, up.oldlogp, up.adv, up.w,
                                    cfg.eps, cfg.loss_scale, loss, out["lse"], out["logp"], out["ratio"],
                                    out["coef"], out["row_loss"])
        torch.cuda.synchronize()
        rel = abs(loss.item() - up.loss.item()) / abs(up.loss.item())
        assert rel < 1e-3, (call, rel)
        for k in OUTS:
            ref = getattr(up, k)[:N]
            err = (out[k] - ref).abs().max().item()
            assert err <= 2e-4 * max(1.0, ref.abs().max().item()), (call, k, err)
