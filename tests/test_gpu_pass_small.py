"""Element-by-element parity of the whole pass (cutoffs, packing, forward, backward) with the
oracle on small workloads that still span several tiles in every GEMM dimension, with
ragged tails. Cutoffs and indices are compared bit-for-bit."""
import numpy as np
import pytest

from synthetic import get_config, make_batch

from gpu_util import check_head, check_prefix, gpu_pass, to_np

pytestmark = pytest.mark.gpu

SMALL = ["tiny", "tiny_bf16", "mid", "mid_f32", "head1.5b_small", "head7b_small"]


@pytest.mark.parametrize("name", SMALL)
def test_pass_matches_oracle(name):
    cfg = get_config(name)
    b, up = gpu_pass(cfg)
    g = to_np(up, up.N)
    N, pk = check_prefix(cfg, b, g)
    assert N == up.N
    stats = check_head(cfg, b, g, pk)
    print(name, N, stats)


@pytest.mark.parametrize("name", ["mid", "tiny"])
def test_full_mode_matches_oracle(name):
    cfg = get_config(name, mode="full")
    b, up = gpu_pass(cfg)
    g = to_np(up, up.N)
    N, pk = check_prefix(cfg, b, g)
    assert N == int(b.L.sum())
    assert np.all(g["w"] == 1.0)
    check_head(cfg, b, g, pk)


@pytest.mark.parametrize("name", ["mid", "mid_f32"])
def test_backward_chunking_and_determinism(name):
    import torch
    cfg = get_config(name)
    b = make_batch(cfg, device="cuda")
    _, whole = gpu_pass(cfg, b, chunk_rows=1 << 20)
    _, chunked = gpu_pass(cfg, b, chunk_rows=128)
    _, again = gpu_pass(cfg, b, chunk_rows=1 << 20)
    N = whole.N
    # dH rows do not depend on the chunking; dW sums chunks in a fixed order
    assert torch.equal(whole.dH[:N], chunked.dH[:N])
    d = (whole.dW - chunked.dW).abs().max().item()
    assert d <= 1e-5 * whole.dW.abs().max().item()
    # bit-identical reruns
    for k in ("lse", "coef", "dH"):
        assert torch.equal(getattr(whole, k)[:N], getattr(again, k)[:N]), k
    assert torch.equal(whole.dW, again.dW) and torch.equal(whole.loss, again.loss)


def test_seeds_and_steps_select_the_cutoff_draw():
    cfg = get_config("tiny_bf16")
    b = make_batch(cfg, device="cuda")
    seen = set()
    for seed, step in ((1, 0), (2, 5), (2**40 + 3, 2**33), (2**64 - 1, 7)):
        _, up = gpu_pass(cfg, b, seed=seed, step=step, grads=False)
        g = to_np(up, up.N)
        check_prefix(cfg, b, g, seed=seed, step=step)
        seen.add(tuple(g["H"]))
    assert len(seen) == 4


@pytest.mark.parametrize("name", ["head7b_small", "mid"])
def test_forward_with_fewer_vocabulary_partials(name):
    # A workspace that holds only a few (max, sum) partials per row makes the forward split the
    # vocabulary into that many ranges; the results must agree with the one-partial-per-tile run.
    import torch
    from paper_2606_29758_gb300 import _binding as B
    cfg = get_config(name)
    b, up = gpu_pass(cfg, grads=False)
    N = up.N
    full = B.ps_lmhead_ppo_fwd_workspace_size(N, cfg.d, cfg.V, up.dcode)
    tiles = (cfg.V + 255) // 256
    for parts in (1, 3, tiles - 1):
        # two 8-byte (max, sum) partials per row and vocabulary range (one per column group of the
        # epilogue): exactly `parts` ranges fit
        small = full - 16 * N * (tiles - parts)
        ws = torch.zeros(small, dtype=torch.uint8, device="cuda")
        outs = {k: torch.empty(N, device="cuda") for k in ("lse", "logp", "ratio", "coef", "row_loss")}
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        D = b.dev
        B.ps_lmhead_ppo_fwd(N, cfg.d, cfg.V, up.dcode, up.hid, D["W"], up.tok, up.oldlogp, up.adv, up.w, cfg.eps,
                            cfg.loss_scale, loss, outs["lse"], outs["logp"], outs["ratio"], outs["coef"],
                            outs["row_loss"], ws)
        torch.cuda.synchronize()
        assert B.ps_workspace_status(ws)[0] == B.PS_OK
        assert abs(loss.item() - up.loss.item()) <= 1e-5 * abs(up.loss.item())
        assert (outs["lse"] - up.lse[:N]).abs().max().item() < 1e-5
    with pytest.raises(B.PsppoError) as e:
        tiny_ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
        B.ps_lmhead_ppo_fwd(N, cfg.d, cfg.V, up.dcode, up.hid, b.dev["W"], up.tok, up.oldlogp, up.adv, up.w,
                            cfg.eps, cfg.loss_scale, loss, outs["lse"], outs["logp"], outs["ratio"], outs["coef"],
                            None, tiny_ws)
    assert e.value.status == B.PS_ERR_WORKSPACE


def test_input_stager_overlapped_copies_give_the_resident_results():
    # Two batches of one shape, copied from pinned host memory through the double-buffered stager
    # while the previous pass runs, must give bit for bit the results of passes on resident inputs.
    import torch
    from paper_2606_29758_gb300 import InputStager
    cfg = get_config("mid")
    b = make_batch(cfg, device="cuda")
    keys = ("q", "L", "R", "tok_full", "oldlogp_full", "hid_full")
    A = {k: b.dev[k] for k in keys}
    Bt = dict(A, R=1.0 - A["R"], tok_full=(A["tok_full"] + 7) % cfg.V, oldlogp_full=A["oldlogp_full"] - 0.01,
              hid_full=A["hid_full"].flip(0).contiguous())
    batches = [A, Bt, A, Bt, Bt]
    ref = []
    for i, X in enumerate(batches):
        _, up = gpu_pass(cfg, b)           # allocate a pass of this shape, then rerun on X
        up.run(X["q"], X["L"], X["R"], X["tok_full"], X["oldlogp_full"], X["hid_full"], b.dev["W"], cfg.seed, i)
        torch.cuda.synchronize()
        ref.append((up.N, up.loss.clone(), up.dH[:up.N].clone(), up.dW.clone()))
    hosts = [{k: v.cpu().pin_memory() for k, v in X.items()} for X in batches]
    _, up = gpu_pass(cfg, b)
    stager = InputStager(hosts[0], device="cuda")
    stream = torch.cuda.current_stream()
    j = stager.stage(hosts[0])
    for i in range(len(batches)):
        X = stager.acquire(j, stream)
        nxt = stager.stage(hosts[i + 1]) if i + 1 < len(batches) else None
        up.run(X["q"], X["L"], X["R"], X["tok_full"], X["oldlogp_full"], X["hid_full"], b.dev["W"], cfg.seed, i)
        stager.release(j, stream)
        torch.cuda.synchronize()
        N, loss, dH, dW = ref[i]
        assert up.N == N
        assert torch.equal(up.loss, loss) and torch.equal(up.dH[:N], dH) and torch.equal(up.dW, dW), i
        j = nxt
    up.check_status()
