"""The vocabulary-parallel head's exchange on gloo ranks (CPU).

Each rank holds one vocabulary shard. It computes its shard's per-row statistics as psppo.h defines
them (m = max_v z log2 e, s = sum_v 2^(z log2 e - m), the chosen logit where the token falls in the
shard, else -inf) and its term of dH (dZ restricted to the shard, times the shard's W), here in float64
from the oracle's logits and the oracle's lse and coef. VocabParallelHead.gather and reduce_dH
exchange them; the statistics merged as the library merges them (m = max_r m_r, s = sum_r s_r
2^(m_r - m), lse = (m + log2 s) ln 2, the chosen logit from its shard) and the summed dH must equal
the oracle's whole-head lse, logp and dH (Eq. 1 through the head of Appendix D).
"""
import os

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

LOG2E = 1.4426950408889634
D, V, N = 24, 50, 40


def _problem():
    rng = np.random.default_rng(11)
    H = rng.standard_normal((N, D))
    W = rng.standard_normal((V, D)) * 0.3
    tok = rng.integers(0, V, N)
    coef = rng.standard_normal(N) * 0.1
    return H, W, tok, coef


def _worker(rank, world, port, out_q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from oracle import lmhead
    from paper_2606_29758_gb300.pipeline import VocabParallelHead, vocab_shards
    H, W, tok, coef = _problem()
    lse = lmhead.logsumexp_rows(lmhead.logits(H, W))
    shards = vocab_shards(V, world)
    vp = VocabParallelHead(shards, N, D, V, torch.float32, device="cpu")
    v0, Vs = shards[rank]
    z = lmhead.logits(H, W[v0:v0 + Vs])                        # [N, Vs]
    x = z * LOG2E
    m = x.max(axis=1)
    s = np.exp2(x - m[:, None]).sum(axis=1)
    inside = (tok >= v0) & (tok < v0 + Vs)
    zt = np.where(inside, z[np.arange(N), np.clip(tok - v0, 0, Vs - 1)], -np.inf)
    vp.stats_all[rank, :N] = torch.from_numpy(np.stack([m, s], axis=1).astype(np.float32))
    vp.ztok_all[rank, :N] = torch.from_numpy(zt.astype(np.float32))
    vp.gather(N, rank)
    # the shard's term of dH: dZ over the shard's columns (one-hot where the token is in the shard)
    dz = -np.exp(z - lse[:, None])
    rows = np.nonzero(inside)[0]
    dz[rows, tok[rows] - v0] += 1.0
    dH = torch.from_numpy(((coef[:, None] * dz) @ W[v0:v0 + Vs]).astype(np.float64))
    vp.reduce_dH(dH)
    if rank == 0:
        out_q.put((vp.stats_all[:, :N].numpy().copy(), vp.ztok_all[:, :N].numpy().copy(), dH.numpy()))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_vocab_shard_statistics_and_dh_exchange_on_gloo_ranks(world):
    from oracle import lmhead
    H, W, tok, coef = _problem()
    zfull = lmhead.logits(H, W)
    lse_ref = lmhead.logsumexp_rows(zfull)
    dH_ref, _ = lmhead.backward(H, W, tok, lse_ref, coef, dw_vocab=[])
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29900 + world * 41 + (os.getpid() % 500)
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    stats, ztok, dH = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    m = stats[:, :, 0].astype(np.float64)
    s = stats[:, :, 1].astype(np.float64)
    M = m.max(axis=0)
    lse = (M + np.log2((s * np.exp2(m - M)).sum(axis=0))) * np.log(2.0)
    np.testing.assert_allclose(lse, lse_ref, rtol=0, atol=2e-6)          # f32-stored statistics
    zt = ztok.max(axis=0)
    np.testing.assert_allclose(zt, zfull[np.arange(N), tok], rtol=1e-6, atol=1e-6)
    assert np.all(np.isfinite(ztok).sum(axis=0) == 1)                   # exactly one shard holds each token
    np.testing.assert_allclose(dH, dH_ref, rtol=1e-12, atol=1e-14)
