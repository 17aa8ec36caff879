"""GB300-native (sm_103a) PS-PPO LM-head update pass.

The computation lives in libpsppo.so (hand-written CUDA, tcgen05 tensor cores, TMA)
behind the C ABI of include/psppo.h; this package is its ctypes binding (same names)
plus UpdatePass, which holds the device buffers of one batch shape in torch, CutoffDesign, which
does the same for the cutoff design upstream of it, InputStager, which copies the next batch
from host memory while the current one runs, and prompt_shard / DataParallelUpdate, one rank's
share of a batch and its step in a data-parallel update, and VocabParallelHead, the head split by
vocabulary rows.
"""
from ._binding import *  # noqa: F401,F403
from ._binding import PsppoError, lib, status_string  # noqa: F401


def __getattr__(name):
    if name in ("UpdatePass", "PassShape", "InputStager", "CutoffDesign", "DesignShape", "PromptShard",
                "prompt_shard", "DataParallelUpdate", "VocabParallelHead", "vocab_shards"):
        from . import pipeline
        return getattr(pipeline, name)
    raise AttributeError(name)
