"""The C-ABI library builds, loads without a GPU, and exports every symbol its headers declare.
Only host-side entry points are called here (status strings, version, workspace sizes)."""
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_29758_gb300 import _build, _binding
    _build.build()
    return _binding.lib()


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names.update(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(ps_\w+)\s*\(", src, flags=re.M))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert {"ps_sample_cutoffs", "ps_pack_prefixes", "ps_lmhead_ppo_fwd", "ps_lmhead_ppo_bwd"} <= names
    for n in sorted(names):
        assert hasattr(lib, n), n


def test_binding_covers_the_headers():
    from paper_2606_29758_gb300 import _binding
    assert set(_binding.EXPORTS) == _declared()
    for n in _binding.EXPORTS:
        assert callable(getattr(_binding, n))


def test_host_only_entry_points(lib):
    from paper_2606_29758_gb300 import _binding as B
    assert B.ps_version() >= 100
    for s in range(8):
        assert isinstance(B.ps_status_string(s), str) and B.ps_status_string(s)
    # forward workspace grows with N; backward workspace with the dZ chunk
    assert B.ps_lmhead_ppo_fwd_workspace_size(1000, 3584, 152064, B.PS_DTYPE_BF16) < \
        B.ps_lmhead_ppo_fwd_workspace_size(2000, 3584, 152064, B.PS_DTYPE_BF16)
    one = B.ps_lmhead_ppo_bwd_workspace_size(100000, 3584, 152064, B.PS_DTYPE_BF16, 128)
    assert one == 256 + 128 * 152064 * 2
    assert B.ps_lmhead_ppo_bwd_workspace_size(100000, 3584, 152064, B.PS_DTYPE_BF16, 1024) == 256 + 1024 * 152064 * 2
    # padded dZ pitch for a vocabulary that is not a multiple of 8
    assert B.ps_lmhead_ppo_bwd_workspace_size(10, 64, 1001, B.PS_DTYPE_F32, 0) == 256 + 128 * 1008 * 4
    assert B.ps_sample_cutoffs_workspace_size(16, 8, 8192) >= 256
    assert B.ps_pack_prefixes_workspace_size(16, 8) >= 256


def test_bad_arguments_are_rejected_before_any_launch(lib):
    import ctypes
    L = lib
    # NULL workspace / bad sizes fail on the host: no device is touched
    assert L.ps_sample_cutoffs(0, 8, 10, None, None, 0, 0, 0, 0, None, None, None, None, 0, None) == 1
    assert L.ps_lmhead_ppo_fwd(-1, 128, 1024, 0, None, None, None, None, None, None, 0.2, 1.0,
                               None, None, None, None, None, None, None, 0, None) == 1
    assert L.ps_lmhead_ppo_bwd(10, 12, 1024, 0, None, None, None, None, None, None, None, 0, None, 0, None) == 1
    assert L.ps_pack_prefixes(1, 1, 1, 8, 7, None, None, None, 1, None, None, None, None, 0,
                              None, None, None, None, None, None, None, None, None,
                              ctypes.POINTER(ctypes.c_int64)(), None, 0, None) == 1


def test_size_limits_and_design_arguments_are_rejected_on_the_host(lib):
    # Every case fails argument checks that run before the first CUDA call (no GPU here).
    import ctypes
    L = lib
    INV = 1
    z = (None,) * 4
    # sampler: group larger than 8192, horizon beyond 2^24, unknown mode
    assert L.ps_sample_cutoffs(1, 8193, 10, *z[:2], 0, 0, 0, 0, None, None, None, None, 0, None) == INV
    assert L.ps_sample_cutoffs(1, 8, (1 << 24) + 1, *z[:2], 0, 0, 0, 0, None, None, None, None, 0, None) == INV
    assert L.ps_sample_cutoffs(1, 8, 10, *z[:2], 0, 0, 0, 7, None, None, None, None, 0, None) == INV
    # head: more rows than int32, a bf16 hidden size that is not a multiple of 8, an empty vocabulary
    fwd = lambda N, d, V, dt: L.ps_lmhead_ppo_fwd(N, d, V, dt, None, None, None, None, None, None, 0.2, 1.0,  # noqa: E731
                                                  None, None, None, None, None, None, None, 0, None)
    assert fwd(1 << 31, 128, 1024, 0) == INV
    assert fwd(10, 100, 1024, 0) == INV
    assert fwd(10, 4, 1024, 0) == INV and fwd(10, 4, 1024, 1) == INV     # d >= 8 for both dtypes
    assert fwd(10, 128, 0, 0) == INV
    assert fwd(10, 128, 1024, 5) == INV
    assert L.ps_lmhead_ppo_bwd(10, 128, 1024, 0, None, None, None, None, None, None, None, 7, None, 0, None) == INV
    assert L.ps_lmhead_ppo_fwd_noalloc(10, 128, 0, 0, None, None, None, None, None, None, 0.2, 1.0,
                                       None, None, None, None, None, None, None) == INV
    assert L.ps_lmhead_ppo_fwd_workspace_size(10, 128, 0, 0) == 0
    # design stage: top-k beyond 16, groups beyond 64 for u_t, unknown strategy, a fixed prefix below 1
    assert L.ps_lmhead_score_proxy(10, 128, 1024, 0, None, None, None, None, None, 17, None, None, None, 0,
                                   None) == INV
    assert L.ps_reward_uncertainty(1, 65, 10, None, None, 16, None, None, None, None, 0, None) == INV
    fake = ctypes.c_void_p(1 << 20)     # never dereferenced: the checks fail first
    assert L.ps_design_cutoffs(1, 8, 10, fake, None, None, 4.0, 9, 0.0, fake, None, None, 0, None) == INV
    assert L.ps_design_cutoffs(1, 8, 10, fake, None, None, 4.0, 4, 0.5, fake, None, None, 0, None) == INV
    assert L.ps_design_cutoffs(1, 8, 10, fake, None, None, 0.0, 3, 0.0, fake, None, None, 0, None) == INV


def test_vocabulary_shard_arguments_are_rejected_on_the_host(lib):
    # The vocabulary-parallel calls check their shard and sizes before any CUDA call (no GPU here).
    L = lib
    INV = 1
    stats = lambda N, d, Vs, v0, dt: L.ps_lmhead_logit_stats(N, d, Vs, v0, dt, None, None, None, None, None,  # noqa: E731
                                                             None, 0, None)
    assert stats(10, 128, 0, 0, 0) == INV           # an empty shard
    assert stats(10, 128, 64, -1, 0) == INV         # a shard before token id 0
    assert stats(-1, 128, 64, 0, 0) == INV
    assert stats(10, 100, 64, 0, 0) == INV          # bf16 hidden size not a multiple of 8
    assert stats(10, 128, 64, 0, 0) == INV          # rows but NULL pointers
    fin = lambda N, S, ld, V: L.ps_lmhead_ppo_fwd_from_stats(N, S, ld, V, None, None, None, None, None, None,  # noqa: E731
                                                             0.2, 1.0, None, None, None, None, None, None, None, 0,
                                                             None)
    assert fin(10, 0, 10, 1024) == INV              # no shard
    assert fin(10, 2, 10, 0) == INV
    assert fin(10, 2, 9, 1024) == INV               # shard stride below the rows
    assert fin(10, 2, 10, 1024) == INV              # NULL loss
    bwd = lambda N, Vs, v0, V: L.ps_lmhead_ppo_bwd_vocab_shard(N, 128, Vs, v0, V, 0, None, None, None, None,  # noqa: E731
                                                               None, None, None, 0, None, 0, None)
    assert bwd(10, 64, 1000, 1024) == INV           # the shard runs past the vocabulary
    assert bwd(10, 64, -5, 1024) == INV
    assert bwd(10, 0, 0, 1024) == INV
    assert L.ps_lmhead_logit_stats_workspace_size(10, 128, 64, 0) == L.ps_lmhead_ppo_fwd_workspace_size(10, 128, 64, 0)
    assert L.ps_lmhead_ppo_fwd_from_stats_workspace_size(1000) >= 256 + 8 * 4


def test_logit_store_layout_and_refusals_on_the_host(lib):
    # The store's size is its layout: [N][ldz] 2-byte values, ldz = V rounded up to 8, then the f32 slice
    # maxima [ceil(V/32)][N] from the next 256-byte boundary. Bad arguments fail before any CUDA call.
    import ctypes
    L = lib
    INV, UNSUP, WS = 1, 2, 3
    assert L.ps_lmhead_logit_store_size(1000, 152064) == 1000 * 152064 * 2 + 4 * 4752 * 1000
    assert L.ps_lmhead_logit_store_size(3, 1001) == 6144 + 4 * 32 * 3          # 3 x 1008 x 2 = 6048 -> 6144
    assert L.ps_lmhead_logit_store_size(0, 1024) == 0
    assert L.ps_lmhead_logit_store_size(-1, 1024) == 0 and L.ps_lmhead_logit_store_size(10, 0) == 0
    assert L.ps_lmhead_ppo_bwd_from_store_workspace_size() == 256
    fake = ctypes.c_void_p(1 << 20)     # 16-byte aligned, never dereferenced: the checks fail first
    p = (fake,) * 6

    def fwd(dt, store, nbytes, d=128, V=1024):
        return L.ps_lmhead_ppo_fwd_store(10, d, V, dt, *p, 0.2, 1.0, fake, fake, fake, fake, fake, None, store,
                                         nbytes, None, 0, None)
    need = L.ps_lmhead_logit_store_size(10, 1024)
    assert fwd(0, None, need) == INV                              # no store
    assert fwd(1, fake, need) == UNSUP                            # f32 head: recompute only
    assert fwd(0, ctypes.c_void_p((1 << 20) + 8), need) == INV    # misaligned store
    assert fwd(0, fake, need - 1) == WS                           # too small
    assert fwd(0, fake, need, d=100) == INV

    def bwd(dt, store, nbytes, flags=0):
        return L.ps_lmhead_ppo_bwd_from_store(10, 128, 1024, dt, *p, store, nbytes, fake, fake, flags, None, 0, None)
    assert bwd(1, fake, need) == UNSUP
    assert bwd(0, None, need) == INV
    assert bwd(0, fake, need, flags=4) == INV                     # unknown flag
    assert bwd(0, fake, need - 1) == WS


def test_vocabulary_shard_store_refusals_on_the_host(lib):
    import ctypes
    L = lib
    INV, UNSUP, WS = 1, 2, 3
    fake = ctypes.c_void_p(1 << 20)
    need = L.ps_lmhead_logit_store_size(10, 64)
    stats = lambda dt, store, nbytes, v0=0: L.ps_lmhead_logit_stats_store(  # noqa: E731
        10, 128, 64, v0, dt, fake, fake, fake, fake, fake, store, nbytes, None, 0, None)
    assert stats(0, None, need) == INV
    assert stats(1, fake, need) == UNSUP
    assert stats(0, fake, need - 1) == WS
    assert stats(0, fake, need, v0=-1) == INV
    bwd = lambda Vs, v0, V, dt=0, nbytes=need: L.ps_lmhead_ppo_bwd_vocab_shard_from_store(  # noqa: E731
        10, 128, Vs, v0, V, dt, fake, fake, fake, fake, fake, fake, fake, nbytes, fake, fake, 0, None, 0, None)
    assert bwd(64, 1000, 1024) == INV           # the shard runs past the vocabulary
    assert bwd(64, 0, 1024, dt=1) == UNSUP
    assert bwd(64, 0, 1024, nbytes=need - 1) == WS
