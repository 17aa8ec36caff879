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
