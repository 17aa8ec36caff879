"""Seeded synthetic inputs for the PS-PPO LM-head update pass.

This package is shared by the tests, the benchmark and the CPU oracle checks. It
draws the rollout batch (lengths, rewards, tokens, hidden states, head weights,
old-policy log-probabilities) and the per-prompt cutoff distribution that the
update pass consumes. It contains none of the update pass itself: no cutoff
sampling, no packing, no advantage normalisation, no loss and no gradient.
"""
from .configs import CONFIGS, Config, get_config  # noqa: F401
from .generate import Batch, make_batch, bf16_bits_to_f32, f32_to_bf16_bits  # noqa: F401
