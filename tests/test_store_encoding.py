"""The logit store's encoding in numpy (no GPU), which fixes the tolerance of its GPU parity test.

The storing forward keeps, for every row and 32-column slice c, e_v = 2^(x_v - m_c) in f16, with
x = z log2 e and m_c the running maximum of the row's x over the columns its vocabulary tile has swept
so far (so e <= 1). The backward forms p_v = e_v 2^(m_c - lse log2 e) and dZ_v = -coef p_v in bf16,
except in the chosen column, which takes coef (1 - exp(logp)). With e at or above 2^-14 (f16
normal), f16 rounding errs by at most 2^-11 relative; below, by at most 2^-25 absolute (half the
subnormal spacing). bf16 rounding errs by at most 2^-8 relative (unit roundoff). So the stored path's
dZ lies within (2^-8 + 2^-11) |dZ| (+ the subnormal floor) of the exact value, the bound
tests/test_gpu_logit_store.py applies; an e kept in bf16 instead would break it.
"""
import numpy as np

LOG2E = 1.4426950408889634


def _bf16(x):
    """Round float32 values to bf16 (nearest, ties to even) and back."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (b + 0x7FFF + ((b >> 16) & 1)) & 0xFFFF0000
    return r.astype(np.uint32).view(np.float32)


def _store_rows(z, tile=256, kind=np.float16):
    """e and the per-slice scale m of rows z [n][V], swept tile by tile (a running maximum reset at
    every 256-column tile, as the forward's per-tile units are), slice by slice inside a tile."""
    n, V = z.shape
    x = (z * LOG2E).astype(np.float32)
    e = np.zeros((n, V), dtype=np.float64)
    m = np.zeros((n, -(-V // 32)), dtype=np.float32)
    for t0 in range(0, V, tile):
        run = np.full(n, -np.inf, dtype=np.float32)
        for c0 in range(t0, min(t0 + tile, V), 32):
            xs = x[:, c0:c0 + 32]
            run = np.maximum(run, xs.max(axis=1))
            m[:, c0 // 32] = run
            e[:, c0:c0 + 32] = np.exp2(xs - run[:, None]).astype(kind).astype(np.float64)
    return e, m


def _dz_from_store(e, m, z, tok, coef):
    V = z.shape[1]
    lse = np.log(np.exp(z - z.max(axis=1, keepdims=True)).sum(axis=1)) + z.max(axis=1)
    f = -coef[:, None] * np.exp2(m[:, np.arange(V) // 32].astype(np.float64) - lse[:, None] * LOG2E)
    dz = _bf16(e * f).astype(np.float64)
    r = np.arange(len(tok))
    logp = z[r, tok] - lse
    dz[r, tok] = _bf16(-coef * np.expm1(logp))
    p = np.exp(z - lse[:, None])
    ref = -coef[:, None] * p
    ref[r, tok] += coef
    return dz, ref, p


def _logits(seed, n=48, V=1000):
    rng = np.random.default_rng(seed)
    z = rng.standard_normal((n, V)) * 1.2
    tok = rng.integers(0, V, n)
    z[:8, :] *= 6.0                              # wide rows: many e in the subnormal range
    z[8:12, tok[8:12]] += 25.0                   # peaked rows: p(o) near 1
    coef = rng.standard_normal(n) * 0.3
    return z, tok, coef


def test_e_is_at_most_one_and_rounds_within_the_f16_bound():
    z, _, _ = _logits(0)
    e, m = _store_rows(z)
    x = z * LOG2E
    exact = np.exp2(x - m[:, np.arange(z.shape[1]) // 32].astype(np.float64))
    assert np.all(e <= 1.0) and np.all(e >= 0.0)
    normal = exact >= 2.0 ** -14
    assert normal.any() and (~normal).any()
    err = np.abs(e - exact)
    assert np.all(err[normal] <= 2.0 ** -11 * exact[normal] * (1 + 1e-6))
    assert np.all(err[~normal] <= 2.0 ** -25 * (1 + 1e-6) + 1e-7 * exact[~normal])


def test_dz_from_the_store_within_the_stated_bound():
    z, tok, coef = _logits(1)
    e, m = _store_rows(z)
    dz, ref, p = _dz_from_store(e, m, z, tok, coef)
    tol = (2.0 ** -8 + 2.0 ** -11) * np.abs(ref) + np.abs(coef)[:, None] * (2.0 ** -22 + 1e-4 * p)
    assert np.all(np.abs(dz - ref) <= tol)
    # the peaked rows' chosen column (1 - p small) keeps its relative accuracy
    r = np.arange(8, 12)
    assert np.all(np.abs(dz[r, tok[r]] - ref[r, tok[r]]) <= 2.0 ** -8 * np.abs(ref[r, tok[r]]) * 1.01)


def test_an_e_kept_in_bf16_breaks_the_bound():
    # the planted mistake: the same store with e rounded to bf16 instead of f16
    z, tok, coef = _logits(2)
    e, m = _store_rows(z, kind=np.float32)
    e = _bf16(e).astype(np.float64)
    dz, ref, p = _dz_from_store(e, m, z, tok, coef)
    tol = (2.0 ** -8 + 2.0 ** -11) * np.abs(ref) + np.abs(coef)[:, None] * (2.0 ** -22 + 1e-4 * p)
    assert np.any(np.abs(dz - ref) > tol)
