"""Data-parallel split of the update pass by prompt groups, on two gloo ranks (CPU).

Advantages are per group, cutoffs are keyed by the global trajectory index and the
loss scale uses the global P*K, so each rank can run its own prompts and the
exchange is a sum of dW (and of the loss). This checks that the shards reproduce
the single-rank result: cutoffs bit-for-bit, loss and dW to rounding.
"""
import os

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle.pipeline import run, widen
from synthetic import get_config, make_batch

CFG = dict(name="tiny", d=24, V=48, P=4, K=3)


def _shard_inputs(b, cfg, rank, world):
    Pp = cfg.P // world
    trajs = slice(rank * Pp * cfg.K, (rank + 1) * Pp * cfg.K)
    off = np.concatenate([[0], np.cumsum(b.L)])
    r0, r1 = off[trajs.start], off[trajs.stop]
    return dict(q=b.q[rank * Pp:(rank + 1) * Pp], L=b.L[trajs], R=b.R[trajs],
                tok=b.tok_full[r0:r1], old=b.oldlogp_full[r0:r1], hid=b.hid_full[r0:r1],
                base=trajs.start)


def _worker(rank, world, port, out_q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    name = CFG["name"]
    cfg = get_config(name, **{k: v for k, v in CFG.items() if k != "name"})
    b = make_batch(cfg)
    s = _shard_inputs(b, cfg, rank, world)
    o = run(s["q"], s["L"], cfg.K, s["R"], s["tok"], s["old"], widen(cfg, s["hid"]), widen(cfg, b.W),
            cfg.eps, cfg.loss_scale, cfg.seed, cfg.step, traj_base=s["base"])
    dW = torch.from_numpy(o["dW"])
    loss = torch.tensor([o["fwd"]["loss"]], dtype=torch.float64)
    H = torch.from_numpy(o["H"]).clone()
    dist.all_reduce(dW)
    dist.all_reduce(loss)
    Hs = [torch.zeros_like(H) for _ in range(world)]
    dist.all_gather(Hs, H)
    if rank == 0:
        out_q.put((dW.numpy(), float(loss[0]), torch.cat(Hs).numpy()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_split_matches_single_rank():
    cfg = get_config(CFG["name"], **{k: v for k, v in CFG.items() if k != "name"})
    b = make_batch(cfg)
    ref = run(b.q, b.L, cfg.K, b.R, b.tok_full, b.oldlogp_full, widen(cfg, b.hid_full), widen(cfg, b.W),
              cfg.eps, cfg.loss_scale, cfg.seed, cfg.step)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + (os.getpid() % 1000)
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    dW, loss, H = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert np.array_equal(H, ref["H"])
    assert loss == pytest.approx(ref["fwd"]["loss"], rel=1e-12)
    np.testing.assert_allclose(dW, ref["dW"], rtol=1e-10, atol=1e-14 * np.abs(ref["dW"]).max())
