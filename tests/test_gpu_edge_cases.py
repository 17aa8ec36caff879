"""Degenerate inputs of the pass, element by element against the oracle: groups of one completion
(zero advantage, so zero gradients), completions of a single token, a vocabulary smaller than one
tile and a vocabulary of one token, the smallest hidden sizes, one prompt with a large group,
and a batch whose every cutoff is H = 0 (nothing to update)."""
from dataclasses import replace

import numpy as np
import pytest

from synthetic import get_config, make_batch

from gpu_util import check_head, check_prefix, gpu_pass, to_np

pytestmark = pytest.mark.gpu

_BASE = get_config("mid")
EDGE = {
    # K = 1: the group's std is 0, every advantage is 0, so are coef, dH, dW and the loss
    "group_of_one": replace(_BASE, name="group_of_one", P=3, K=1, len_lo=1, len_hi=40, d=64, V=300),
    # every completion is one token long (T_max = 1), head narrower than one K block
    "one_token": replace(_BASE, name="one_token", P=2, K=4, len_lo=1, len_hi=1, d=8, V=5),
    # a vocabulary of one token: softmax = 1, log p = 0, dZ = 0
    "vocab_one": replace(_BASE, name="vocab_one", P=2, K=4, len_lo=1, len_hi=30, d=16, V=1),
    # f32 at the smallest hidden size the library takes (d = 8), three tokens
    "f32_d8": replace(_BASE, name="f32_d8", dtype="f32", P=2, K=4, len_lo=1, len_hi=50, d=8, V=3),
    # one prompt, 64 completions, lengths from 1 to 200 (many ragged tails)
    "wide_group": replace(_BASE, name="wide_group", P=1, K=64, len_lo=1, len_hi=200, d=136, V=520),
}


@pytest.mark.parametrize("name", list(EDGE))
def test_degenerate_shapes_match_oracle(name):
    cfg = EDGE[name]
    b, up = gpu_pass(cfg, chunk_rows=128)
    g = to_np(up, up.N)
    N, pk = check_prefix(cfg, b, g)
    assert N == up.N
    stats = check_head(cfg, b, g, pk)
    print(name, N, stats)
    if name == "group_of_one":
        assert np.all(g["adv"] == 0) and np.all(g["coef"] == 0)
        assert g["loss"] == 0.0 and np.all(g["dH"] == 0) and np.all(g["dW"] == 0)
    if name == "vocab_one":
        assert np.abs(g["logp"]).max() < 1e-6
    if name == "one_token":
        assert np.all(g["n"] == 1) and np.all(g["w"] == 1)


def test_all_cutoffs_zero_gives_an_empty_pass():
    # Masses that sum to 0 in the H = 0 mode: every completion keeps no token (Pr(H = 0) = 1).
    import torch
    from oracle.cutoffs import sample_cutoffs
    from paper_2606_29758_gb300 import PS_MODE_TRUNC_ZERO, PassShape, UpdatePass
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    q = np.zeros_like(b.q)
    D = dict(b.dev)
    D["q"] = torch.zeros_like(D["q"])
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, 128),
                    eps=cfg.eps, loss_scale=cfg.loss_scale, mode=PS_MODE_TRUNC_ZERO)
    up.loss.fill_(float("nan"))
    up.dW.fill_(float("nan"))
    N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    torch.cuda.synchronize()
    up.check_status()
    H, n, _ = sample_cutoffs(q, b.L, cfg.K, cfg.seed, cfg.step, mode="trunc_zero")
    assert N == 0 and np.all(H == 0) and np.all(n == 0)
    assert np.array_equal(up.H.cpu().numpy(), H) and np.array_equal(up.n.cpu().numpy(), n)
    assert np.all(up.cu_seqlens.cpu().numpy() == 0)
    assert up.loss.item() == 0.0
    assert bool((up.dW == 0).all())      # overwritten with zeros, not left as it was


@pytest.mark.parametrize("name,over", [
    # the largest group the sampler takes (K = 8192, its shared-memory scan), short completions
    ("max_group", dict(P=1, K=8192, len_lo=1, len_hi=4, d=8, V=5)),
    # a horizon of 2^20 steps (two completions of up to a million tokens), a tiny head; seed 3
    # draws different rewards for the two, so the advantages (and gradients) are not zero
    ("long_horizon", dict(P=1, K=2, len_lo=1 << 19, len_hi=1 << 20, d=8, V=7, seed=3)),
])
def test_largest_groups_and_horizons_match_oracle(name, over):
    cfg = replace(_BASE, name=name, **over)
    b, up = gpu_pass(cfg, chunk_rows=1 << 16)
    g = to_np(up, up.N)
    N, pk = check_prefix(cfg, b, g)
    assert N == up.N and b.T_max == int(b.L.max())
    stats = check_head(cfg, b, g, pk)
    print(name, N, b.T_max, stats)
    assert np.any(g["adv"] != 0) and np.abs(g["dW"]).max() > 0
