"""Pins for the oracle's cutoff sampler and weights (Section 3.2, Appendices B-C)."""
import math

import numpy as np
import pytest

from oracle.cutoffs import (ONE62, cumulative_masses, cutoff_from_uniform, inverse_survival_weights,
                            sample_cutoffs, survival, xi)
from synthetic.generate import beta_masses


def _masses(T, seed=0):
    rng = np.random.default_rng(seed)
    a, b = rng.uniform(0.5, 3.0, size=2)
    return beta_masses(T, a, b)


def test_budget_identity_expected_cutoff_equals_sum_of_xi():
    # Section 3.3: sum_t t (xi_t - xi_{t+1}) = E[H], and telescoping gives sum_t xi_t.
    for T in (1, 2, 7, 100, 1000):
        q = _masses(T, T)
        S = survival(q)
        EH_num = sum((h + 1) * int(m) for h, m in enumerate(q))      # 2^62 * E[H]
        assert sum(S) == EH_num                                         # exact integers
        xs = list(S) + [0]
        assert sum((t + 1) * (xs[t] - xs[t + 1]) for t in range(T)) == EH_num


def test_survival_is_monotone_and_starts_at_one():
    q = _masses(300)
    x = xi(q)
    assert x[0] == 1.0
    assert np.all(np.diff(x) <= 0) and np.all(x > 0)


def test_cutoff_boundaries():
    q = np.array([5, 0, 3, ONE62 - 8], dtype=np.uint64)
    U = cumulative_masses(q)
    assert cutoff_from_uniform(U, 0) == 1
    assert cutoff_from_uniform(U, 4) == 1
    assert cutoff_from_uniform(U, 5) == 3          # zero-mass bucket 2 is skipped
    assert cutoff_from_uniform(U, 7) == 3
    assert cutoff_from_uniform(U, 8) == 4
    assert cutoff_from_uniform(U, ONE62 - 1) == 4


def test_weights_invert_survival():
    q = _masses(500, 3)
    w = inverse_survival_weights(q)
    x = xi(q)
    reach = x > 0
    np.testing.assert_allclose(w[reach] * x[reach], 1.0, rtol=1e-15)
    assert w[0] == 1.0


def test_full_mode_is_identity():
    L = np.array([5, 9, 3, 7], dtype=np.int32)
    q = np.zeros((2, 9), dtype=np.uint64)
    q[:, 0] = ONE62
    H, n, w = sample_cutoffs(q, L, 2, seed=3, step=1, mode="full")
    assert np.array_equal(H, L) and np.array_equal(n, L) and np.all(w == 1.0)


def test_bad_masses_rejected():
    q = np.zeros((1, 4), dtype=np.uint64)
    q[0, 0] = ONE62 - 1
    with pytest.raises(ValueError):
        sample_cutoffs(q, np.array([4], dtype=np.int32), 1, seed=0, step=0)


@pytest.mark.slow
def test_sampling_statistics_match_xi():
    # One prompt, T = 40, many independent draws (steps): the empirical survival and
    # E[(I_t/xi_t - 1)^2] = 1/xi_t - 1 (Appendix C) hold within sampling error.
    T, M = 40, 6000
    q = _masses(T, 11)
    x = xi(q)
    L = np.full(1, T, dtype=np.int32)
    Hs = np.array([sample_cutoffs(q[None], L, 1, seed=5, step=s)[0][0] for s in range(M)])
    surv = np.array([(Hs >= t).mean() for t in range(1, T + 1)])
    se = np.sqrt(x * (1 - x) / M) + 1e-12
    assert np.all(np.abs(surv - x) <= 4.5 * se + 1e-9)
    # Pearson chi-square over the cutoff values with expected count >= 5
    p = np.array([int(m) / ONE62 for m in q])
    obs = np.bincount(Hs, minlength=T + 1)[1:]
    keep = p * M >= 5
    chi2 = (((obs[keep] - p[keep] * M) ** 2) / (p[keep] * M)).sum()
    dof = keep.sum() - 1
    assert chi2 < dof + 5 * math.sqrt(2 * dof)
    # mean cutoff vs sum of xi (CLT bound)
    EH = x.sum()
    sdH = math.sqrt(sum(((h + 1) - EH) ** 2 * p[h] for h in range(T)))
    assert abs(Hs.mean() - EH) < 4.5 * sdH / math.sqrt(M)
    # Appendix C: E[(I/xi - 1)^2] = 1/xi - 1
    for t in (1, 5, 10, 20):
        I = (Hs >= t).astype(np.float64)
        emp = ((I / x[t - 1] - 1.0) ** 2).mean()
        exact = 1.0 / x[t - 1] - 1.0
        sd = math.sqrt(max(exact * (1 + exact), 1e-30) / M) * 3 + 1e-12
        assert abs(emp - exact) < 4.5 * sd + 1e-9


def test_sharded_draws_match_whole_batch():
    # cutoffs are keyed by the global trajectory index: two shards reproduce the whole batch
    rng = np.random.default_rng(1)
    P, K = 4, 3
    L = rng.integers(5, 30, size=P * K).astype(np.int32)
    q = np.zeros((P, 30), dtype=np.uint64)
    for p in range(P):
        q[p, :L[p * K:(p + 1) * K].max()] = _masses(int(L[p * K:(p + 1) * K].max()), p)
    H, n, w = sample_cutoffs(q, L, K, seed=9, step=4)
    H0, n0, w0 = sample_cutoffs(q[:2], L[:6], K, seed=9, step=4, traj_base=0)
    H1, n1, w1 = sample_cutoffs(q[2:], L[6:], K, seed=9, step=4, traj_base=6)
    assert np.array_equal(np.concatenate([H0, H1]), H)
    assert np.array_equal(np.concatenate([w0, w1]), w)
