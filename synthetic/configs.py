"""The five synthetic workloads of the LM-head PS-PPO update pass, plus small
test shapes.

Each workload is a rollout batch of P prompts x K completions (B = P*K
trajectories), a per-prompt cutoff distribution, and an LM head of hidden size d
and vocabulary V. The shapes mirror the paper's math setting (K = 8 completions
per prompt, Section 4 and Appendix I; Qwen-sized heads with V ~ 152k) without
using any of its data.
"""
from dataclasses import dataclass, replace
from typing import Optional, Tuple


@dataclass(frozen=True)
class Config:
    name: str
    P: int                      # prompts
    K: int                      # completions per prompt (group size)
    len_law: str                # "uniform" | "lognormal"
    len_lo: int                 # lengths clipped to [len_lo, len_hi]
    len_hi: int
    len_median: Optional[int]   # lognormal median (None for uniform)
    d: int                      # hidden size
    V: int                      # vocabulary size
    dtype: str                  # "f32" | "bf16" (storage of hidden states and W)
    beta_a: Tuple[float, float]  # per-prompt Beta(a, b) cutoff law, a ~ U[lo, hi]
    beta_b: Tuple[float, float]
    eps: float = 0.2            # PPO clip range
    mode: str = "trunc"         # "trunc" (sampled cutoffs) | "full" (cutoff = length, w = 1)
    adv_mode: int = 1           # 1: (R - mean) / (std + 1e-6); 0: R - mean
    seed: int = 0
    step: int = 0
    lognormal_sigma: float = 0.5
    w_std: float = 0.02
    oldlogp_noise: float = 0.05

    @property
    def B(self) -> int:
        return self.P * self.K

    @property
    def loss_scale(self) -> float:
        # 1/K per prompt (Eq. full_update_G) averaged over the P prompts.
        return 1.0 / (self.P * self.K)


_BETA = ((0.5, 3.0), (0.5, 3.0))

CONFIGS = {
    "tiny": Config("tiny", P=2, K=4, len_law="uniform", len_lo=32, len_hi=256, len_median=None,
                   d=128, V=1024, dtype="f32", beta_a=_BETA[0], beta_b=_BETA[1]),
    "1.5b": Config("1.5b", P=32, K=8, len_law="lognormal", len_lo=64, len_hi=4096, len_median=1024,
                   d=1536, V=151936, dtype="bf16", beta_a=_BETA[0], beta_b=_BETA[1]),
    "7b": Config("7b", P=16, K=8, len_law="lognormal", len_lo=128, len_hi=8192, len_median=2048,
                 d=3584, V=152064, dtype="bf16", beta_a=_BETA[0], beta_b=_BETA[1]),
    "long": Config("long", P=8, K=16, len_law="uniform", len_lo=8192, len_hi=16384, len_median=None,
                   d=3584, V=152064, dtype="bf16", beta_a=(0.5, 1.0), beta_b=(2.0, 4.0)),
}
CONFIGS["full"] = replace(CONFIGS["7b"], name="full", mode="full")

# Small shapes for parity tests: several tiles in every GEMM dimension, ragged tails.
CONFIGS["tiny_bf16"] = replace(CONFIGS["tiny"], name="tiny_bf16", dtype="bf16")
CONFIGS["mid"] = Config("mid", P=2, K=4, len_law="uniform", len_lo=40, len_hi=300, len_median=None,
                        d=392, V=2000, dtype="bf16", beta_a=_BETA[0], beta_b=_BETA[1])
CONFIGS["head7b_small"] = Config("head7b_small", P=1, K=4, len_law="uniform", len_lo=60, len_hi=150,
                                 len_median=None, d=3584, V=152064, dtype="bf16",
                                 beta_a=_BETA[0], beta_b=_BETA[1])
CONFIGS["head1.5b_small"] = Config("head1.5b_small", P=1, K=4, len_law="uniform", len_lo=60, len_hi=150,
                                   len_median=None, d=1536, V=151936, dtype="bf16",
                                   beta_a=_BETA[0], beta_b=_BETA[1])
CONFIGS["mid_f32"] = replace(CONFIGS["mid"], name="mid_f32", dtype="f32")
# The 7B-shaped head on two prompts (about 25k packed rows): a small case for profiling.
CONFIGS["7b_p2"] = replace(CONFIGS["7b"], name="7b_p2", P=2)
# The 7B-shaped head on one group of four (about 7k packed rows): a capture of a few GB of device memory.
CONFIGS["7b_p1k4"] = replace(CONFIGS["7b"], name="7b_p1k4", P=1, K=4)


def get_config(name: str, **overrides) -> Config:
    cfg = CONFIGS[name]
    return replace(cfg, **overrides) if overrides else cfg
