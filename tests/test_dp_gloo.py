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


class _OraclePass:
    """A CPU stand-in for UpdatePass with the same calls, computed by the oracle (test
    infrastructure): it lets the library's data-parallel orchestration (prompt_shard,
    DataParallelUpdate) run on gloo ranks without a GPU."""

    def __init__(self, cfg, W, loss_scale):
        self.cfg, self.W, self.loss_scale = cfg, W, loss_scale
        self.dW = None
        self.loss = torch.zeros(1, dtype=torch.float64)

    def sample(self, q, L, seed, step, traj_base=0):
        from oracle.cutoffs import sample_cutoffs
        self.H, self.n, self.w_tab = sample_cutoffs(q, L, self.cfg.K, seed, step, traj_base=traj_base)

    def pack(self, L, R, tok_full, oldlogp_full, hid_full):
        from oracle.pack import group_advantages, pack_prefixes
        A = group_advantages(R, self.cfg.K, self.cfg.adv_mode)
        self.pk = pack_prefixes(L, self.n, self.cfg.K, self.w_tab, A, tok_full, oldlogp_full, hid_full)
        return self.pk["N"]

    def forward(self, W):
        from oracle import lmhead
        pk = self.pk
        self.f = lmhead.forward(widen(self.cfg, pk["hid"]), self.W, pk["tok"], pk["oldlogp"], pk["adv"], pk["w"],
                                self.cfg.eps, self.loss_scale)
        self.loss = torch.tensor([self.f["loss"]], dtype=torch.float64)

    def backward(self, W):
        from oracle import lmhead
        pk = self.pk
        _, dW = lmhead.backward(widen(self.cfg, pk["hid"]), self.W, pk["tok"], self.f["lse"], self.f["coef"])
        self.dW = torch.from_numpy(dW)


def _dp_worker(rank, world, port, out_q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2606_29758_gb300.pipeline import DataParallelUpdate, prompt_shard
    cfg = get_config(CFG["name"], **{k: v for k, v in CFG.items() if k != "name"})
    b = make_batch(cfg)
    sh = prompt_shard(cfg.P, cfg.K, b.L, world, rank)
    dpu = DataParallelUpdate(_OraclePass(cfg, widen(cfg, b.W), cfg.loss_scale), traj_base=sh.k0)
    assert dpu.world() == world
    n = dpu.run(b.q[sh.p0:sh.p1], b.L[sh.k0:sh.k1], b.R[sh.k0:sh.k1], b.tok_full[sh.o0:sh.o1],
                b.oldlogp_full[sh.o0:sh.o1], b.hid_full[sh.o0:sh.o1], None, cfg.seed, cfg.step)
    rows = torch.tensor([n])
    dist.all_reduce(rows)
    Hs = [None] * world                          # shards may hold different numbers of prompts
    dist.all_gather_object(Hs, dpu.up.H)
    if rank == 0:
        out_q.put((dpu.up.dW.numpy(), float(dpu.up.loss[0]), np.concatenate(Hs), int(rows[0])))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_data_parallel_update_orchestration_on_gloo_ranks(world):
    # the library's rank step (DataParallelUpdate over prompt_shard), each rank an oracle pass over its
    # shard: the summed dW and loss, the gathered cutoffs and the total rows equal the whole batch's
    cfg = get_config(CFG["name"], **{k: v for k, v in CFG.items() if k != "name"})
    b = make_batch(cfg)
    ref = run(b.q, b.L, cfg.K, b.R, b.tok_full, b.oldlogp_full, widen(cfg, b.hid_full), widen(cfg, b.W),
              cfg.eps, cfg.loss_scale, cfg.seed, cfg.step)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29700 + world * 37 + (os.getpid() % 500)
    procs = [ctx.Process(target=_dp_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    dW, loss, H, rows = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert np.array_equal(H, ref["H"]) and rows == ref["pack"]["N"]
    assert loss == pytest.approx(ref["fwd"]["loss"], rel=1e-12)
    np.testing.assert_allclose(dW, ref["dW"], rtol=1e-10, atol=1e-14 * np.abs(ref["dW"]).max())
