"""Parity at the workloads' full sizes, in the launch configuration the benchmark times.

Cutoffs, weights, advantages and every packing index/row are compared bit-for-bit with
the oracle over the whole batch. The head is compared on sampled rows the oracle can
evaluate one by one (random rows, the largest weights, and rows where the clip binds):
lse, logp, ratio, coef, row loss and the dH row. For dW, which sums over every row,
two properties that hold at any size are checked: sum_v dW[v, :] = 0 (the softmax score
e_o - p sums to zero over the vocabulary) within the bound set by the bf16 rounding of
dZ, and loss = sum of row losses. Then dW itself: the backward runs again over all N rows
of the oracle's packed batch with the oracle's lse and coef on the sampled rows and coef = 0
on every other row (whose dZ row is then zero), so dW = sum over the sampled rows, which the
oracle evaluates on every vocabulary row that a sampled row chose plus 512 random ones.
"""
import numpy as np
import pytest
import torch

from synthetic import get_config, make_batch

from gpu_util import GRAD_MAXREL, check_head, oracle_prefix

pytestmark = pytest.mark.gpu

CHUNK = 65536   # the benchmark's backward chunk


def _pull(t, N):
    return t[:N].cpu().numpy()


@pytest.mark.parametrize("name", ["1.5b", "7b", "long", "full"])
def test_full_size(name):
    from paper_2606_29758_gb300 import PS_MODE_FULL, PS_MODE_TRUNC, PassShape, UpdatePass
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    D = b.dev
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, CHUNK),
                    eps=cfg.eps, loss_scale=cfg.loss_scale,
                    mode=PS_MODE_FULL if cfg.mode == "full" else PS_MODE_TRUNC)
    N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    torch.cuda.synchronize()
    up.check_status()

    H, n, w_tab, A, pk = oracle_prefix(cfg, b)
    assert N == pk["N"]
    assert np.array_equal(up.H.cpu().numpy(), H) and np.array_equal(up.n.cpu().numpy(), n)
    g_w = up.w_tab.cpu().numpy()
    fin = np.isfinite(w_tab)
    assert np.array_equal(g_w[fin], w_tab[fin].astype(np.float32)) and np.all(np.isinf(g_w[~fin]))
    assert np.array_equal(up.cu_seqlens.cpu().numpy(), pk["cu_seqlens"])
    for k in ("src_row", "row_traj", "row_pos", "tok"):
        assert np.array_equal(_pull(getattr(up, k), N), pk[k]), k
    assert np.array_equal(_pull(up.oldlogp, N), pk["oldlogp"].astype(np.float32))
    assert np.array_equal(_pull(up.w, N), pk["w"].astype(np.float32))
    assert np.array_equal(_pull(up.adv, N), pk["adv"].astype(np.float32))
    hid = up.hid[:N].view(torch.int16).cpu().numpy().view(np.uint16)
    assert np.array_equal(hid, pk["hid"])

    # sampled rows for the head
    rng = np.random.default_rng(1234)
    coef = _pull(up.coef, N)
    adv = pk["adv"]
    bind = np.nonzero((coef == 0) & (adv != 0))[0]
    heavy = np.argsort(pk["w"])[-16:]
    rows = np.unique(np.concatenate([rng.choice(N, size=min(N, 768), replace=False), heavy,
                                     bind[:64], [0, N - 1]])).astype(np.int64)
    g = {"lse": _pull(up.lse, N), "logp": _pull(up.logp, N), "ratio": _pull(up.ratio, N), "coef": coef,
         "row_loss": _pull(up.row_loss, N), "w": _pull(up.w, N)}
    dH = np.zeros((N, cfg.d), dtype=np.float32)
    sel = torch.from_numpy(rows).cuda()
    dH[rows] = up.dH[sel].cpu().numpy()
    g["dH"] = dH
    rep = {}
    stats = check_head(cfg, b, g, pk, rows=rows, report=rep)
    print(name, N, len(rows), stats)

    # loss = sum of row losses (the row losses are checked above)
    total = float(up.row_loss[:N].double().sum().item())
    assert abs(up.loss.item() - total) <= 1e-5 * abs(up.loss.item()) + 1e-12

    # sum over the vocabulary of dW vanishes up to the bf16 rounding of dZ:
    # |sum_v dZ~_iv| <= 2^-8 |coef_i|  =>  |sum_v dW[v, c]| <= 2^-8 sum_i |coef_i| |h_ic| (+ f32 sums)
    colsum = up.dW.double().sum(dim=0)
    hf = up.hid[:N].float()
    bound = (up.coef[:N].abs()[:, None] * hf.abs()).double().sum(dim=0) * 2.0 ** -8
    ratio = (colsum.abs() / (1.5 * bound + 1e-6 * up.dW.abs().max().double())).max().item()
    assert ratio < 1.0, ratio
    assert torch.isfinite(up.dW).all() and torch.isfinite(up.dH[:N]).all()

    # dW at full size: same N, chunking and kernels; only the sampled rows carry a coefficient
    from oracle import lmhead
    from oracle.pipeline import widen
    from paper_2606_29758_gb300 import _binding as B
    idx, lse_o, coef_o = rep["oracle_rows"], rep["oracle_lse"], rep["oracle_coef"]
    lse32 = np.zeros(N, dtype=np.float32)
    coef32 = np.zeros(N, dtype=np.float32)
    lse32[idx], coef32[idx] = lse_o.astype(np.float32), coef_o.astype(np.float32)
    hid_o = torch.from_numpy(pk["hid"].view(np.int16)).cuda().view(torch.bfloat16)
    tok_o = torch.from_numpy(pk["tok"].astype(np.int32)).cuda()
    dH2 = torch.empty(N, cfg.d, dtype=torch.float32, device="cuda")
    dW2 = torch.empty(cfg.V, cfg.d, dtype=torch.float32, device="cuda")
    up.ws_bwd.zero_()
    B.ps_lmhead_ppo_bwd(N, cfg.d, cfg.V, up.dcode, hid_o, D["W"], tok_o, torch.from_numpy(lse32).cuda(),
                        torch.from_numpy(coef32).cuda(), dH2, dW2, B.PS_DW_OVERWRITE, up.ws_bwd)
    torch.cuda.synchronize()
    up.check_status()
    vocab = np.unique(np.concatenate([pk["tok"][idx], rng.choice(cfg.V, size=512, replace=False)]))
    _, dW_ref = lmhead.backward(widen(cfg, pk["hid"][idx]), widen(cfg, b.W), pk["tok"][idx],
                                lse32[idx].astype(np.float64), coef32[idx].astype(np.float64),
                                dh_rows=[], dw_vocab=vocab)
    got = dW2[torch.from_numpy(vocab).cuda()].double().cpu().numpy()
    err = float(np.abs(got - dW_ref).max() / np.abs(dW_ref).max())
    print(name, "dW over", len(idx), "rows,", len(vocab), "vocab rows: max-rel", err)
    assert err < GRAD_MAXREL, err
    # every other row's dZ is zero, so the unsampled rows of dH vanish
    others = torch.ones(N, dtype=torch.bool, device="cuda")
    others[torch.from_numpy(idx).cuda()] = False
    assert float(dH2[others].abs().max().item()) == 0.0
