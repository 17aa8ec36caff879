"""Pins for advantages and packing, and the full-cutoff invariant of the whole oracle pass."""
import math

import numpy as np
import pytest

from oracle import lmhead
from oracle.pack import group_advantages, pack_prefixes
from oracle.pipeline import run, widen
from synthetic import get_config, make_batch


def test_advantage_closed_form():
    # rewards [1, 0, 0, 0]: mean 1/4, population std sqrt(3)/4
    A = group_advantages(np.array([1, 0, 0, 0], dtype=np.float32), 4, 1)
    sd = math.sqrt(3) / 4
    np.testing.assert_allclose(A, np.array([0.75, -0.25, -0.25, -0.25]) / (sd + 1e-6), rtol=1e-15)
    A0 = group_advantages(np.array([1, 0, 0, 0], dtype=np.float32), 4, 0)
    np.testing.assert_allclose(A0, [0.75, -0.25, -0.25, -0.25], rtol=1e-15)


def test_advantage_degenerate_group_is_zero():
    # Section 4 (rollouts K): all-correct or all-wrong groups carry no signal
    A = group_advantages(np.array([1, 1, 1, 0, 0, 0], dtype=np.float32), 3, 1)
    assert np.all(A == 0.0)


def test_advantage_group_moments():
    R = np.random.default_rng(0).random(64).astype(np.float32)
    A = group_advantages(R, 8, 1).reshape(8, 8)
    np.testing.assert_allclose(A.mean(axis=1), 0.0, atol=1e-12)
    np.testing.assert_allclose(A.std(axis=1), 1.0, rtol=1e-4)


def test_packing_layout():
    L = np.array([3, 5, 2, 4])
    n = np.array([2, 5, 1, 3])
    w_tab = np.arange(10, dtype=np.float64).reshape(2, 5) + 1
    tok = np.arange(100, 114)
    old = -np.arange(14, dtype=np.float64)
    hid = np.arange(14 * 2, dtype=np.float64).reshape(14, 2)
    pk = pack_prefixes(L, n, 2, w_tab, np.array([.1, .2, .3, .4]), tok, old, hid)
    assert pk["N"] == 11
    assert list(pk["cu_seqlens"]) == [0, 2, 7, 8, 11]
    assert list(pk["src_row"]) == [0, 1, 3, 4, 5, 6, 7, 8, 10, 11, 12]
    assert list(pk["row_traj"]) == [0, 0, 1, 1, 1, 1, 1, 2, 3, 3, 3]
    assert list(pk["row_pos"]) == [1, 2, 1, 2, 3, 4, 5, 1, 1, 2, 3]
    assert list(pk["w"]) == [1, 2, 1, 2, 3, 4, 5, 6, 6, 7, 8]
    assert list(pk["adv"]) == [.1, .1, .2, .2, .2, .2, .2, .3, .4, .4, .4]
    assert np.array_equal(pk["tok"], tok[pk["src_row"]])
    assert np.array_equal(pk["hid"], hid[pk["src_row"]])


@pytest.mark.parametrize("name", ["tiny", "tiny_bf16"])
def test_full_cutoff_reduces_to_untruncated_clipped_surrogate(name):
    # With H = L and w = 1 the pass is Eq. 1 summed over every completion token,
    # 1/K per prompt, averaged over prompts -- evaluated here directly per completion.
    cfg = get_config(name, d=32, V=64)
    b = make_batch(cfg)
    hid, W = widen(cfg, b.hid_full), widen(cfg, b.W)
    out = run(b.q, b.L, cfg.K, b.R, b.tok_full, b.oldlogp_full, hid, W, cfg.eps, cfg.loss_scale,
              cfg.seed, cfg.step, mode="full", grads=False)
    A = group_advantages(b.R, cfg.K, 1)
    J = 0.0
    off = 0
    for p in range(cfg.P):
        Jp = 0.0
        for j in range(cfg.K):
            k = p * cfg.K + j
            rows = np.arange(off, off + int(b.L[k]))
            off += int(b.L[k])
            z = hid[rows] @ W.T
            m = z.max(axis=1)
            lp = z[np.arange(rows.size), b.tok_full[rows]] - (m + np.log(np.exp(z - m[:, None]).sum(axis=1)))
            rho = np.exp(lp - b.oldlogp_full[rows].astype(np.float64))
            Jp += np.minimum(rho * A[k], np.clip(rho, 1 - cfg.eps, 1 + cfg.eps) * A[k]).sum()
        J += Jp / cfg.K
    J /= cfg.P
    assert out["fwd"]["loss"] == pytest.approx(-J, rel=1e-12)
    assert out["pack"]["N"] == int(b.L.sum())
    assert np.array_equal(out["pack"]["hid"], hid)


def test_truncated_pass_rows_and_weights():
    cfg = get_config("tiny", d=16, V=32)
    b = make_batch(cfg)
    out = run(b.q, b.L, cfg.K, b.R, b.tok_full, b.oldlogp_full, widen(cfg, b.hid_full), widen(cfg, b.W),
              cfg.eps, cfg.loss_scale, cfg.seed, cfg.step, grads=False)
    n = out["n"]
    assert np.all(n >= 1) and np.all(n <= b.L) and out["pack"]["N"] == int(n.sum())
    assert np.all(out["pack"]["w"] >= 1.0)
    assert lmhead is not None
