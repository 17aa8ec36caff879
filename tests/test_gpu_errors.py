"""Device-side checks report through the workspace status word; nothing faults.
Bad data is made on the host: masses that do not sum to 2^62, a length out of range, a
capacity that is too small, a token id outside the vocabulary, a workspace that is too small."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _B():
    from paper_2606_29758_gb300 import _binding as B
    return B


def _sample(q, L, K, mode=0):
    B = _B()
    P, T = q.shape
    H = torch.empty(P * K, dtype=torch.int32, device="cuda")
    n = torch.empty_like(H)
    w = torch.empty(P, T, dtype=torch.float32, device="cuda")
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    B.ps_sample_cutoffs(P, K, T, torch.from_numpy(q.view(np.int64)).cuda(), torch.from_numpy(L).cuda(),
                        3, 1, 0, mode, H, n, w, ws)
    return B.ps_workspace_status(ws), H, n, w


def test_bad_masses_set_bad_pmf():
    B = _B()
    q = np.zeros((2, 8), dtype=np.uint64)
    q[0, 0] = 1 << 62
    q[1, :] = 1 << 59          # sums to 2^62 exactly
    (rc, bits), *_ = _sample(q, np.array([8, 8, 8, 8], dtype=np.int32), 2)
    assert rc == B.PS_OK and bits == 0
    q[1, 3] += 1               # one too many
    (rc, bits), *_ = _sample(q, np.array([8, 8, 8, 8], dtype=np.int32), 2)
    assert rc == B.PS_ERR_DEVICE_DATA and bits & B.PS_DEV_BAD_PMF
    q[1, 3] = np.uint64((1 << 63) + 5)   # a single mass above 2^62 (the scan saturates, no wrap)
    (rc, bits), *_ = _sample(q, np.array([8, 8, 8, 8], dtype=np.int32), 2)
    assert rc == B.PS_ERR_DEVICE_DATA and bits & B.PS_DEV_BAD_PMF


def test_bad_length_is_reported():
    B = _B()
    q = np.zeros((1, 8), dtype=np.uint64)
    q[0, 7] = 1 << 62
    (rc, bits), *_ = _sample(q, np.array([8, 9], dtype=np.int32), 2)
    assert rc == B.PS_ERR_DEVICE_DATA and bits & B.PS_DEV_BAD_LENGTH
    (rc, bits), *_ = _sample(q, np.array([0, 3], dtype=np.int32), 2, mode=B.PS_MODE_FULL)
    assert bits & B.PS_DEV_BAD_LENGTH


def test_capacity_and_bad_token_and_small_workspace():
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    from synthetic import get_config, make_batch
    B = _B()
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    D = b.dev
    # capacity one row short of the full length: fine for the truncated pass only if N fits
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, 16, torch.bfloat16), eps=cfg.eps)
    up.sample(D["q"], D["L"], cfg.seed, cfg.step)
    N = up.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"])
    rc, bits = B.ps_workspace_status(up.ws_pack)
    assert rc == B.PS_ERR_CAPACITY and bits & B.PS_DEV_CAPACITY
    assert up.cu_seqlens[-1].item() == N and N > 16   # the count is still reported
    # a token id outside the vocabulary
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16), eps=cfg.eps)
    tok_bad = D["tok_full"].clone()
    tok_bad[0] = cfg.V
    up.sample(D["q"], D["L"], cfg.seed, cfg.step)
    up.pack(D["L"], D["R"], tok_bad, D["oldlogp_full"], D["hid_full"])
    up.forward(D["W"])
    rc, bits = B.ps_workspace_status(up.ws_fwd)
    assert rc == B.PS_ERR_DEVICE_DATA and bits & B.PS_DEV_BAD_TOKEN
    assert torch.isnan(up.logp[0]).item()
    # a workspace smaller than required is refused on the host
    small = torch.empty(1024, dtype=torch.uint8, device="cuda")
    with pytest.raises(B.PsppoError) as e:
        B.ps_lmhead_ppo_fwd(up.N, cfg.d, cfg.V, B.PS_DTYPE_BF16, up.hid, D["W"], up.tok, up.oldlogp, up.adv, up.w,
                            0.2, 1.0, up.loss, up.lse, up.logp, up.ratio, up.coef, None, small)
    assert e.value.status == B.PS_ERR_WORKSPACE


def test_non_finite_inputs_stay_in_their_rows():
    # A NaN hidden state poisons its own row, the loss and the dW sum over rows, and nothing else;
    # an old log-prob of +inf gives ratio 0 and a finite loss. No status bit is set: non-finite
    # inputs are passed through, not detected.
    from synthetic import get_config, make_batch
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    D = b.dev

    def run(hid, old):
        up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, 128),
                        eps=cfg.eps, loss_scale=cfg.loss_scale)
        up.run(D["q"], D["L"], D["R"], D["tok_full"], old, hid, D["W"], cfg.seed, cfg.step)
        torch.cuda.synchronize()
        up.check_status()
        return up

    clean = run(D["hid_full"], D["oldlogp_full"])
    N = clean.N
    hid = D["hid_full"].clone()
    hid[0, 5] = float("nan")                 # token 1 of completion 0: always packed, as row 0
    bad = run(hid, D["oldlogp_full"])
    assert bad.N == N and torch.isnan(bad.lse[0]) and torch.isnan(bad.row_loss[0])
    assert torch.isnan(bad.loss).all()                 # as in the definition: min and clip keep a NaN
    for k in ("lse", "logp", "ratio", "coef"):
        assert torch.equal(getattr(bad, k)[1:N], getattr(clean, k)[1:N]), k
    assert torch.equal(bad.dH[1:N], clean.dH[1:N]) and torch.isnan(bad.dH[0]).any()
    old = D["oldlogp_full"].clone()
    old[0] = float("inf")
    inf_run = run(D["hid_full"], old)
    assert float(inf_run.ratio[0]) == 0.0 and torch.isfinite(inf_run.loss).all()
    assert torch.isfinite(inf_run.dW).all() and torch.isfinite(inf_run.dH[:N]).all()


def test_non_finite_design_weight_sets_its_bit():
    B = _B()
    from synthetic import get_config
    from synthetic.generate import draw_design_inputs, draw_lengths
    cfg = get_config("mid")
    L = draw_lengths(cfg)
    gamma, u = draw_design_inputs(cfg, L)
    gamma[3] = np.nan
    T = int(L.max())
    q = torch.empty(cfg.P, T, dtype=torch.int64, device="cuda")
    ws = torch.zeros(B.ps_design_cutoffs_workspace_size(cfg.P, cfg.K, T), dtype=torch.uint8, device="cuda")
    B.ps_design_cutoffs(cfg.P, cfg.K, T, torch.from_numpy(L).cuda(), torch.from_numpy(gamma).cuda(),
                        torch.from_numpy(u).cuda(), 40.0, B.PS_DESIGN_OPTIMIZED, 0.0, q, None, ws)
    rc, bits = B.ps_workspace_status(ws)
    assert rc == B.PS_ERR_DEVICE_DATA and bits & B.PS_DEV_NONFINITE
    # the same inputs with the NaN removed are accepted
    gamma[3] = 1.0
    B.ps_design_cutoffs(cfg.P, cfg.K, T, torch.from_numpy(L).cuda(), torch.from_numpy(gamma).cuda(),
                        torch.from_numpy(u).cuda(), 40.0, B.PS_DESIGN_OPTIMIZED, 0.0, q, None, ws)
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
