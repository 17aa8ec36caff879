"""Stored values of the oracle's Tiny pass (tests/golden/tiny_oracle_pass.json, written by
tests/golden/make_golden.py from oracle/ only; the paper prints no worked numeric example).

CPU: the oracle still reproduces them (a regression record of the oracle). GPU: the CUDA path on
the same host-generated inputs matches them within the path's tolerances, without running the
oracle."""
import json
import os

import numpy as np
import pytest

from oracle.pipeline import run, widen
from synthetic import get_config, make_batch
from synthetic.generate import to_device

GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "tiny_oracle_pass.json")


def _gold():
    with open(GOLD) as fh:
        return json.load(fh)


def test_oracle_reproduces_the_stored_pass():
    g = _gold()
    cfg = get_config("tiny")
    b = make_batch(cfg)
    o = run(b.q, b.L, cfg.K, b.R, b.tok_full, b.oldlogp_full, widen(cfg, b.hid_full), widen(cfg, b.W),
            cfg.eps, cfg.loss_scale, cfg.seed, cfg.step)
    assert [int(x) for x in o["H"]] == g["H"] and int(o["pack"]["N"]) == g["N"]
    rows, vocab = g["rows"], g["vocab"]
    assert o["fwd"]["loss"] == pytest.approx(g["loss"], rel=1e-12)
    np.testing.assert_allclose(o["fwd"]["lse"][rows], g["lse"], rtol=1e-12)
    np.testing.assert_allclose(o["fwd"]["coef"][rows], g["coef"], rtol=1e-12)
    np.testing.assert_allclose(o["dH"][rows].sum(axis=1), g["dH_row_sums"], rtol=1e-9, atol=1e-15)
    np.testing.assert_allclose(o["dW"][vocab].sum(axis=1), g["dW_row_sums"], rtol=1e-9, atol=1e-15)
    assert np.abs(o["dW"]).sum() == pytest.approx(g["dW_abs_sum"], rel=1e-12)


@pytest.mark.gpu
def test_cuda_path_matches_the_stored_pass():
    import torch
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    g = _gold()
    cfg = get_config("tiny")
    b = make_batch(cfg)
    D = to_device(b, "cuda")
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.float32),
                    eps=cfg.eps, loss_scale=cfg.loss_scale)
    N = up.run(D["q"], D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"], D["W"], cfg.seed, cfg.step)
    torch.cuda.synchronize()
    up.check_status()
    assert up.H.cpu().tolist() == g["H"] and N == g["N"]
    rows = torch.tensor(g["rows"], device="cuda")
    assert abs(up.loss.item() - g["loss"]) <= 1e-3 * abs(g["loss"])
    np.testing.assert_allclose(up.lse[rows].cpu().numpy(), g["lse"], rtol=2e-6)
    np.testing.assert_allclose(up.coef[rows].cpu().numpy(), g["coef"], rtol=2e-4)
    dW = up.dW.double().cpu().numpy()
    assert abs(np.abs(dW).sum() - g["dW_abs_sum"]) <= 2e-2 * g["dW_abs_sum"]
