"""Seeded generators for one synthetic rollout batch.

Every quantity comes from its own numpy PCG64 stream keyed by
(seed, stream id[, block]), so any block of hidden-state rows can be redrawn on
its own and the large arrays are drawn in parallel. The recipe:

* lengths L_k: uniform integers on [lo, hi], or round(exp(ln(median) + 0.5 z))
  clipped to [lo, hi] (lognormal);
* per prompt p, a_p ~ U[a_lo, a_hi] and b_p ~ U[b_lo, b_hi]; the cutoff pmf over
  h = 1..T_p (T_p = longest completion of the group) is the Beta(a_p, b_p) mass
  of ((h-1)/T_p, h/T_p], quantised to non-negative integers that sum to 2^62
  (floor of mass * 2^62; the remainder, of either sign, goes to the largest
  bucket, lowest index on ties);
* rewards R_k ~ Bernoulli(0.5); tokens uniform on [0, V);
* hidden states h ~ N(0, 1) over [sum L, d]; W ~ N(0, 0.02) over [V, d], stored
  [V, d] (vocabulary-major, like an LM head weight); both rounded
  to bfloat16 (round to nearest even) for bf16 workloads;
* old-policy log-probabilities: the log-probability of each token under the
  rounded (hidden, W), plus N(0, 0.05) noise.

The last item needs the token log-probability of every completion position; it
is a fixture recipe evaluated with plain torch/numpy matmuls and is never used
as an expected value. Both the CUDA path and the oracle receive the resulting
array as an input.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field
from typing import Dict, Optional

import numpy as np

from .configs import Config

ONE62 = 1 << 62

_S_LEN, _S_BETA, _S_REW, _S_TOK, _S_HID, _S_W, _S_NOISE = range(7)
_ROW_BLOCK = 8192


def _rng(cfg_seed: int, *keys: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([cfg_seed, *keys]))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round finite float32 values to bfloat16 (nearest, ties to even); returns raw uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of raw bfloat16 bits to float32."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def draw_lengths(cfg: Config) -> np.ndarray:
    g = _rng(cfg.seed, _S_LEN)
    if cfg.len_law == "uniform":
        L = g.integers(cfg.len_lo, cfg.len_hi + 1, size=cfg.B)
    elif cfg.len_law == "lognormal":
        z = g.standard_normal(cfg.B)
        L = np.rint(np.exp(math.log(cfg.len_median) + cfg.lognormal_sigma * z))
        L = np.clip(L, cfg.len_lo, cfg.len_hi)
    else:
        raise ValueError(cfg.len_law)
    return L.astype(np.int32)


def beta_masses(T: int, a: float, b: float) -> np.ndarray:
    """Integer masses q[h-1], h = 1..T, of Beta(a, b) on the cells ((h-1)/T, h/T]; sum exactly 2^62."""
    from scipy.special import betainc
    edges = np.arange(T + 1, dtype=np.float64) / T
    cdf = betainc(a, b, edges)
    m = np.clip(np.diff(cdf), 0.0, None)
    m = m / m.sum()
    q = np.floor(m * float(ONE62)).astype(np.uint64)
    rem = ONE62 - int(q.sum(dtype=np.uint64))   # |rem| is at most ~T + 2^62 * (fp64 rounding of the sum)
    i = int(np.argmax(q))
    q[i] = np.uint64(int(q[i]) + rem)
    assert int(q.sum(dtype=np.uint64)) == ONE62
    return q


def draw_cutoff_pmf(cfg: Config, L: np.ndarray) -> (np.ndarray, np.ndarray):
    """Per-prompt integer cutoff masses [P, T_max] (zero beyond the group's longest completion)."""
    g = _rng(cfg.seed, _S_BETA)
    a = g.uniform(cfg.beta_a[0], cfg.beta_a[1], size=cfg.P)
    b = g.uniform(cfg.beta_b[0], cfg.beta_b[1], size=cfg.P)
    T_max = int(L.max())
    q = np.zeros((cfg.P, T_max), dtype=np.uint64)
    for p in range(cfg.P):
        Tp = int(L[p * cfg.K:(p + 1) * cfg.K].max())
        q[p, :Tp] = beta_masses(Tp, float(a[p]), float(b[p]))
    return q, np.stack([a, b], axis=1)


def _parallel_rows(total: int, fn, out: np.ndarray) -> None:
    blocks = [(i, min(i + _ROW_BLOCK, total)) for i in range(0, total, _ROW_BLOCK)]
    workers = max(1, min(len(blocks), os.cpu_count() or 1))
    with ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(lambda blk: fn(blk[0] // _ROW_BLOCK, blk[0], blk[1], out), blocks))


def draw_matrix(cfg: Config, stream: int, rows: int, cols: int, std: float) -> np.ndarray:
    """N(0, std^2) matrix [rows, cols]: float32, or bf16 bits (uint16) for bf16 workloads."""
    bf16 = cfg.dtype == "bf16"
    out = np.empty((rows, cols), dtype=np.uint16 if bf16 else np.float32)

    def fill(bi, r0, r1, o):
        x = _rng(cfg.seed, stream, bi).standard_normal((r1 - r0, cols), dtype=np.float32)
        if std != 1.0:
            x *= np.float32(std)
        o[r0:r1] = f32_to_bf16_bits(x) if bf16 else x

    _parallel_rows(rows, fill, out)
    return out


def hidden_rows(cfg: Config, rows: np.ndarray) -> np.ndarray:
    """Redraw selected rows of the hidden-state matrix (identical to the full draw)."""
    rows = np.asarray(rows, dtype=np.int64)
    out = np.empty((rows.size, cfg.d), dtype=np.uint16 if cfg.dtype == "bf16" else np.float32)
    for bi in np.unique(rows // _ROW_BLOCK):
        r0 = int(bi) * _ROW_BLOCK
        sel = np.nonzero(rows // _ROW_BLOCK == bi)[0]
        hi = int(rows[sel].max()) + 1
        x = _rng(cfg.seed, _S_HID, int(bi)).standard_normal((hi - r0, cfg.d), dtype=np.float32)
        x = x[rows[sel] - r0]
        out[sel] = f32_to_bf16_bits(x) if cfg.dtype == "bf16" else x
    return out


def as_f32(cfg: Config, m: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(m) if cfg.dtype == "bf16" else m


@dataclass
class Batch:
    """One synthetic rollout batch on the host (numpy), optionally mirrored on a torch device."""
    cfg: Config
    L: np.ndarray            # int32 [B]
    q: np.ndarray            # uint64 [P, T_max]
    beta_ab: np.ndarray      # float64 [P, 2]
    R: np.ndarray            # float32 [B]
    tok_full: np.ndarray     # int32 [sum L]
    hid_full: np.ndarray     # bf16 bits (uint16) or float32 [sum L, d]
    W: np.ndarray            # bf16 bits (uint16) or float32 [V, d]
    oldlogp_full: np.ndarray  # float32 [sum L]
    dev: Dict[str, object] = field(default_factory=dict)

    @property
    def T_max(self) -> int:
        return int(self.q.shape[1])

    @property
    def total_len(self) -> int:
        return int(self.L.sum())


def _token_logprobs_numpy(hid32: np.ndarray, W32: np.ndarray, tok: np.ndarray) -> np.ndarray:
    out = np.empty(tok.shape[0], dtype=np.float64)
    W64 = W32.astype(np.float64)
    for r0 in range(0, tok.shape[0], 256):
        z = hid32[r0:r0 + 256].astype(np.float64) @ W64.T
        m = z.max(axis=1, keepdims=True)
        lse = m[:, 0] + np.log(np.exp(z - m).sum(axis=1))
        out[r0:r0 + 256] = z[np.arange(z.shape[0]), tok[r0:r0 + 256]] - lse
    return out


def _token_logprobs_torch(hid, W, tok, chunk: int = 8192):
    import torch
    out = torch.empty(tok.shape[0], dtype=torch.float32, device=hid.device)
    for r0 in range(0, tok.shape[0], chunk):
        z = torch.matmul(hid[r0:r0 + chunk], W.t()).float()
        out[r0:r0 + chunk] = z.gather(1, tok[r0:r0 + chunk, None].long())[:, 0] - torch.logsumexp(z, dim=1)
    return out


def make_batch(cfg: Config, device: Optional[str] = None) -> Batch:
    """Draw one batch. With a torch device, also place the inputs there (under .dev)."""
    L = draw_lengths(cfg)
    q, ab = draw_cutoff_pmf(cfg, L)
    R = (_rng(cfg.seed, _S_REW).random(cfg.B) < 0.5).astype(np.float32)
    total = int(L.sum())
    tok = _rng(cfg.seed, _S_TOK).integers(0, cfg.V, size=total).astype(np.int32)
    hid = draw_matrix(cfg, _S_HID, total, cfg.d, 1.0)
    W = draw_matrix(cfg, _S_W, cfg.V, cfg.d, cfg.w_std)
    noise = _rng(cfg.seed, _S_NOISE).standard_normal(total).astype(np.float64) * cfg.oldlogp_noise
    b = Batch(cfg, L, q, ab, R, tok, hid, W, np.zeros(total, np.float32))
    if device is None:
        lp = _token_logprobs_numpy(as_f32(cfg, hid), as_f32(cfg, W), tok)
        b.oldlogp_full = (lp + noise).astype(np.float32)
        return b
    import torch
    b.dev = to_device(b, device)
    lp = _token_logprobs_torch(b.dev["hid_full"], b.dev["W"], b.dev["tok_full"]).double().cpu().numpy()
    b.oldlogp_full = (lp + noise).astype(np.float32)
    b.dev["oldlogp_full"] = torch.from_numpy(b.oldlogp_full).to(device)
    return b


def torch_matrix(cfg: Config, m: np.ndarray):
    import torch
    t = torch.from_numpy(m.view(np.int16) if cfg.dtype == "bf16" else m)
    return t.view(torch.bfloat16) if cfg.dtype == "bf16" else t


def to_device(b: Batch, device: str) -> Dict[str, object]:
    import torch
    d = {
        "L": torch.from_numpy(b.L).to(device),
        "q": torch.from_numpy(b.q.view(np.int64)).to(device),
        "R": torch.from_numpy(b.R).to(device),
        "tok_full": torch.from_numpy(b.tok_full).to(device),
        "hid_full": torch_matrix(b.cfg, b.hid_full).to(device),
        "W": torch_matrix(b.cfg, b.W).to(device),
        "oldlogp_full": torch.from_numpy(b.oldlogp_full).to(device),
    }
    return d


_S_GAMMA, _S_UNC = 7, 8


def draw_design_inputs(cfg: Config, L: np.ndarray):
    """Inputs of the cutoff-design step: a positive per-token score gamma in completion order
    (a decaying trend times lognormal noise, so that adjacent timesteps often violate the
    monotone order) and a reward-uncertainty proxy u [P, T_max] on [0.02, 0.25]."""
    g = _rng(cfg.seed, _S_GAMMA)
    total = int(L.sum())
    t = np.concatenate([np.arange(int(n), dtype=np.float64) for n in L])
    gamma = (cfg.d * (1.0 + 3.0 * np.exp(-t / 200.0)) * np.exp(0.7 * g.standard_normal(total))).astype(np.float32)
    u = _rng(cfg.seed, _S_UNC).uniform(0.02, 0.25, size=(cfg.P, int(L.max()))).astype(np.float32)
    return gamma, u
