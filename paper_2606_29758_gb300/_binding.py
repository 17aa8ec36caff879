"""ctypes binding of libpsppo (include/psppo.h, include/psppo_diag.h).

Argument marshalling only: torch tensors become device pointers, the current torch
CUDA stream becomes the cudaStream_t, and a non-zero ps_status becomes a
PsppoError. Every step of the computation runs in the library's kernels; there is
no fallback, and importing this module without the built library raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libpsppo.so")

PS_OK, PS_ERR_INVALID_ARG, PS_ERR_UNSUPPORTED, PS_ERR_WORKSPACE, PS_ERR_CAPACITY, \
    PS_ERR_DEVICE_DATA, PS_ERR_TIMEOUT, PS_ERR_CUDA = range(8)
PS_MODE_TRUNC, PS_MODE_FULL, PS_MODE_TRUNC_ZERO = 0, 1, 2
PS_DTYPE_BF16, PS_DTYPE_F32 = 0, 1
PS_ADV_CENTERED, PS_ADV_GROUP_NORM = 0, 1
PS_DW_OVERWRITE, PS_DW_ACCUMULATE, PS_DH_ACCUMULATE = 0, 1, 2
PS_DEV_BAD_PMF, PS_DEV_BAD_LENGTH, PS_DEV_CAPACITY, PS_DEV_BAD_TOKEN, PS_DEV_TIMEOUT, PS_DEV_NONFINITE = \
    1, 2, 4, 8, 16, 32

EXPORTS = [
    "ps_status_string", "ps_version", "ps_workspace_status",
    "ps_sample_cutoffs_workspace_size", "ps_sample_cutoffs",
    "ps_pack_prefixes_workspace_size", "ps_pack_prefixes",
    "ps_lmhead_ppo_fwd_workspace_size", "ps_lmhead_ppo_fwd",
    "ps_lmhead_ppo_bwd_workspace_size", "ps_lmhead_ppo_bwd",
    "ps_lmhead_logit_stats_workspace_size", "ps_lmhead_logit_stats",
    "ps_lmhead_ppo_fwd_from_stats_workspace_size", "ps_lmhead_ppo_fwd_from_stats", "ps_lmhead_ppo_bwd_vocab_shard",
    "ps_lmhead_logit_store_size", "ps_lmhead_ppo_fwd_store", "ps_lmhead_ppo_bwd_from_store_workspace_size",
    "ps_lmhead_ppo_bwd_from_store", "ps_lmhead_logit_stats_store", "ps_lmhead_ppo_bwd_vocab_shard_from_store",
    "ps_diag_gemm_bf16", "ps_diag_wait_timeout", "ps_lmhead_ppo_fwd_noalloc",
    "ps_lmhead_score_proxy_workspace_size", "ps_lmhead_score_proxy",
    "ps_design_cutoffs_workspace_size", "ps_design_cutoffs",
    "ps_reward_uncertainty_workspace_size", "ps_reward_uncertainty", "ps_binarize_rewards",
]
PS_DESIGN_OPTIMIZED, PS_DESIGN_HEURISTIC, PS_DESIGN_UNIFORM, PS_DESIGN_TIME_PRIOR, PS_DESIGN_FIXED = range(5)


__all__ = EXPORTS + [
    "PsppoError", "lib", "status_string", "dtype_code", "LIB_PATH",
    "PS_OK", "PS_ERR_INVALID_ARG", "PS_ERR_UNSUPPORTED", "PS_ERR_WORKSPACE", "PS_ERR_CAPACITY",
    "PS_ERR_DEVICE_DATA", "PS_ERR_TIMEOUT", "PS_ERR_CUDA", "PS_MODE_TRUNC", "PS_MODE_FULL", "PS_MODE_TRUNC_ZERO",
    "PS_DTYPE_BF16", "PS_DTYPE_F32", "PS_ADV_CENTERED", "PS_ADV_GROUP_NORM", "PS_DW_OVERWRITE",
    "PS_DW_ACCUMULATE", "PS_DH_ACCUMULATE", "PS_DEV_BAD_PMF", "PS_DEV_BAD_LENGTH", "PS_DEV_CAPACITY", "PS_DEV_BAD_TOKEN",
    "PS_DEV_TIMEOUT", "PS_DEV_NONFINITE", "PS_DESIGN_OPTIMIZED", "PS_DESIGN_HEURISTIC", "PS_DESIGN_UNIFORM",
    "PS_DESIGN_TIME_PRIOR", "PS_DESIGN_FIXED",
]


class PsppoError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


_lib: Optional[ctypes.CDLL] = None

_vp, _sz, _i32, _i64, _u64, _f64 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_int64, \
    ctypes.c_uint64, ctypes.c_double

_SIGS = {
    "ps_status_string": (ctypes.c_char_p, [_i32]),
    "ps_version": (_i32, []),
    "ps_workspace_status": (_i32, [_vp, _vp, ctypes.POINTER(ctypes.c_uint32)]),
    "ps_sample_cutoffs_workspace_size": (_sz, [_i32, _i32, _i32]),
    "ps_sample_cutoffs": (_i32, [_i32, _i32, _i32, _vp, _vp, _u64, _u64, _i64, _i32, _vp, _vp, _vp, _vp, _sz, _vp]),
    "ps_pack_prefixes_workspace_size": (_sz, [_i32, _i32]),
    "ps_pack_prefixes": (_i32, [_i32, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _i64,
                                _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, ctypes.POINTER(ctypes.c_int64),
                                _vp, _sz, _vp]),
    "ps_lmhead_ppo_fwd_workspace_size": (_sz, [_i64, _i32, _i32, _i32]),
    "ps_lmhead_ppo_fwd": (_i32, [_i64, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _f64, _f64,
                                 _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "ps_lmhead_ppo_bwd_workspace_size": (_sz, [_i64, _i32, _i32, _i32, _i64]),
    "ps_lmhead_ppo_bwd": (_i32, [_i64, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _vp, _sz, _vp]),
    "ps_lmhead_logit_stats_workspace_size": (_sz, [_i64, _i32, _i32, _i32]),
    "ps_lmhead_logit_stats": (_i32, [_i64, _i32, _i32, _i64, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "ps_lmhead_ppo_fwd_from_stats_workspace_size": (_sz, [_i64]),
    "ps_lmhead_ppo_fwd_from_stats": (_i32, [_i64, _i32, _i64, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _f64, _f64, _vp, _vp,
                                            _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "ps_lmhead_ppo_bwd_vocab_shard": (_i32, [_i64, _i32, _i32, _i64, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                             _i32, _vp, _sz, _vp]),
    "ps_lmhead_logit_store_size": (_sz, [_i64, _i32]),
    "ps_lmhead_ppo_fwd_store": (_i32, [_i64, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _f64, _f64,
                                       _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _sz, _vp]),
    "ps_lmhead_ppo_bwd_from_store_workspace_size": (_sz, []),
    "ps_lmhead_ppo_bwd_from_store": (_i32, [_i64, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _vp,
                                            _i32, _vp, _sz, _vp]),
    "ps_lmhead_logit_stats_store": (_i32, [_i64, _i32, _i32, _i64, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _sz,
                                           _vp]),
    "ps_lmhead_ppo_bwd_vocab_shard_from_store": (_i32, [_i64, _i32, _i32, _i64, _i32, _i32, _vp, _vp, _vp, _vp, _vp,
                                                        _vp, _vp, _sz, _vp, _vp, _i32, _vp, _sz, _vp]),
    "ps_diag_gemm_bf16": (_i32, [_i32, _i32, _i32, _i32, _i32, _vp, _i64, _vp, _i64, _vp, _i64, _i32, _i32, _vp, _sz,
                                 _vp]),
    "ps_diag_wait_timeout": (_i32, [_u64, _vp, _sz, _vp]),
    "ps_lmhead_score_proxy_workspace_size": (_sz, [_i64, _i32, _i32, _i32, _i32]),
    "ps_lmhead_score_proxy": (_i32, [_i64, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _sz,
                                     _vp]),
    "ps_reward_uncertainty_workspace_size": (_sz, [_i32, _i32]),
    "ps_reward_uncertainty": (_i32, [_i32, _i32, _i32, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _sz, _vp]),
    "ps_binarize_rewards": (_i32, [_i32, _vp, _u64, _u64, _i64, _vp, _vp]),
    "ps_design_cutoffs_workspace_size": (_sz, [_i32, _i32, _i32]),
    "ps_design_cutoffs": (_i32, [_i32, _i32, _i32, _vp, _vp, _vp, _f64, _i32, _f64, _vp, _vp, _vp, _sz, _vp]),
    "ps_lmhead_ppo_fwd_noalloc": (_i32, [_i64, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _f64, _f64,
                                         _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
}


def lib() -> ctypes.CDLL:
    """Load libpsppo.so from the package directory (built by __graft_entry__.build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"libpsppo.so is not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().ps_status_string(int(status)).decode()


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr()


def _stream(stream=None) -> Optional[int]:
    if stream is not None:
        return int(stream) if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def _check(rc: int, where: str) -> None:
    if rc != PS_OK:
        raise PsppoError(rc, where)


def _nbytes(t) -> int:
    return t.numel() * t.element_size()


def dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return PS_DTYPE_BF16
    if t.dtype == torch.float32:
        return PS_DTYPE_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


# ----------------------------------------------------------------------------- entry points
def ps_status_string(status: int) -> str:
    return status_string(status)


def ps_version() -> int:
    return lib().ps_version()


def ps_workspace_status(ws, stream=None):
    """Synchronise the stream and return (ps_status, raw PS_DEV_* bits) of a workspace."""
    bits = ctypes.c_uint32(0)
    rc = lib().ps_workspace_status(_ptr(ws), _stream(stream), ctypes.byref(bits))
    return rc, bits.value


def ps_sample_cutoffs_workspace_size(P: int, K: int, T_max: int) -> int:
    return lib().ps_sample_cutoffs_workspace_size(P, K, T_max)


def ps_sample_cutoffs(P, K, T_max, q, L, seed, step, traj_base, mode, H, n, w_tab, ws, stream=None):
    rc = lib().ps_sample_cutoffs(P, K, T_max, _ptr(q), _ptr(L), seed & (2**64 - 1), step & (2**64 - 1),
                                 traj_base, mode, _ptr(H), _ptr(n), _ptr(w_tab), _ptr(ws), _nbytes(ws),
                                 _stream(stream))
    _check(rc, "ps_sample_cutoffs")


def ps_pack_prefixes_workspace_size(P: int, K: int) -> int:
    return lib().ps_pack_prefixes_workspace_size(P, K)


def ps_pack_prefixes(P, K, T_max, d, dtype, L, n, R, adv_mode, w_tab, tok_full, oldlogp_full, hid_full,
                     capacity, cu_seqlens, src_row, row_traj, row_pos, tok, oldlogp, w, adv, hid_packed, ws,
                     return_num_rows=True, stream=None) -> Optional[int]:
    nrows = ctypes.c_int64(-1)
    rc = lib().ps_pack_prefixes(P, K, T_max, d, dtype, _ptr(L), _ptr(n), _ptr(R), adv_mode, _ptr(w_tab),
                                _ptr(tok_full), _ptr(oldlogp_full), _ptr(hid_full), capacity, _ptr(cu_seqlens),
                                _ptr(src_row), _ptr(row_traj), _ptr(row_pos), _ptr(tok), _ptr(oldlogp), _ptr(w),
                                _ptr(adv), _ptr(hid_packed), ctypes.byref(nrows) if return_num_rows else None,
                                _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_pack_prefixes")
    return int(nrows.value) if return_num_rows else None


def ps_lmhead_ppo_fwd_workspace_size(N: int, d: int, V: int, dtype: int) -> int:
    return lib().ps_lmhead_ppo_fwd_workspace_size(N, d, V, dtype)


def ps_lmhead_ppo_fwd(N, d, V, dtype, Hpk, W, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp, ratio,
                      coef, row_loss, ws, stream=None):
    rc = lib().ps_lmhead_ppo_fwd(N, d, V, dtype, _ptr(Hpk), _ptr(W), _ptr(tok), _ptr(oldlogp), _ptr(adv), _ptr(w),
                                 float(eps), float(loss_scale), _ptr(loss), _ptr(lse), _ptr(logp), _ptr(ratio),
                                 _ptr(coef), _ptr(row_loss), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_ppo_fwd")


def ps_lmhead_ppo_fwd_noalloc(N, d, V, dtype, Hpk, W, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp, ratio,
                              coef, row_loss, stream=None):
    """The forward with the library's static device scratch instead of a workspace, for
    callers that cannot allocate device memory (see include/psppo.h)."""
    rc = lib().ps_lmhead_ppo_fwd_noalloc(N, d, V, dtype, _ptr(Hpk), _ptr(W), _ptr(tok), _ptr(oldlogp), _ptr(adv),
                                         _ptr(w), float(eps), float(loss_scale), _ptr(loss), _ptr(lse), _ptr(logp),
                                         _ptr(ratio), _ptr(coef), _ptr(row_loss), _stream(stream))
    _check(rc, "ps_lmhead_ppo_fwd_noalloc")


def ps_lmhead_score_proxy_workspace_size(N: int, d: int, V: int, dtype: int, topk: int = 0) -> int:
    return lib().ps_lmhead_score_proxy_workspace_size(N, d, V, dtype, topk)


def ps_lmhead_score_proxy(N, d, V, dtype, Hrows, W, tok, gamma, logp, ws, topk=0, top_idx=None, top_prob=None,
                          stream=None):
    rc = lib().ps_lmhead_score_proxy(N, d, V, dtype, _ptr(Hrows), _ptr(W), _ptr(tok), _ptr(gamma), _ptr(logp), topk,
                                     _ptr(top_idx), _ptr(top_prob), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_score_proxy")


def ps_reward_uncertainty_workspace_size(P: int, K: int) -> int:
    return lib().ps_reward_uncertainty_workspace_size(P, K)


def ps_reward_uncertainty(P, K, T_max, L, R, topk, top_idx, top_prob, u, ws, stream=None):
    rc = lib().ps_reward_uncertainty(P, K, T_max, _ptr(L), _ptr(R), topk, _ptr(top_idx), _ptr(top_prob), _ptr(u),
                                     _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_reward_uncertainty")


def ps_binarize_rewards(B, R, seed, step, y, traj_base=0, stream=None):
    rc = lib().ps_binarize_rewards(B, _ptr(R), seed, step, traj_base, _ptr(y), _stream(stream))
    _check(rc, "ps_binarize_rewards")


def ps_design_cutoffs_workspace_size(P: int, K: int, T_max: int) -> int:
    return lib().ps_design_cutoffs_workspace_size(P, K, T_max)


def ps_design_cutoffs(P, K, T_max, L, gamma_full, u, budget, strategy, param, q, xi, ws, stream=None):
    rc = lib().ps_design_cutoffs(P, K, T_max, _ptr(L), _ptr(gamma_full), _ptr(u), float(budget), int(strategy),
                                 float(param), _ptr(q), _ptr(xi), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_design_cutoffs")


def ps_lmhead_ppo_bwd_workspace_size(N: int, d: int, V: int, dtype: int, chunk_rows: int = 0) -> int:
    return lib().ps_lmhead_ppo_bwd_workspace_size(N, d, V, dtype, chunk_rows)


def ps_lmhead_ppo_bwd(N, d, V, dtype, Hpk, W, tok, lse, coef, dH, dW, flags, ws, stream=None):
    rc = lib().ps_lmhead_ppo_bwd(N, d, V, dtype, _ptr(Hpk), _ptr(W), _ptr(tok), _ptr(lse), _ptr(coef), _ptr(dH),
                                 _ptr(dW), flags, _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_ppo_bwd")


def ps_lmhead_logit_stats_workspace_size(N: int, d: int, Vs: int, dtype: int) -> int:
    return lib().ps_lmhead_logit_stats_workspace_size(N, d, Vs, dtype)


def ps_lmhead_logit_stats(N, d, Vs, v0, dtype, Hpk, W_shard, tok, stats, ztok, ws, stream=None):
    rc = lib().ps_lmhead_logit_stats(N, d, Vs, v0, dtype, _ptr(Hpk), _ptr(W_shard), _ptr(tok), _ptr(stats),
                                     _ptr(ztok), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_logit_stats")


def ps_lmhead_ppo_fwd_from_stats_workspace_size(N: int) -> int:
    return lib().ps_lmhead_ppo_fwd_from_stats_workspace_size(N)


def ps_lmhead_ppo_fwd_from_stats(N, S, ld, V, stats, ztok, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp,
                                 ratio, coef, row_loss, ws, stream=None):
    rc = lib().ps_lmhead_ppo_fwd_from_stats(N, S, ld, V, _ptr(stats), _ptr(ztok), _ptr(tok), _ptr(oldlogp), _ptr(adv),
                                            _ptr(w), float(eps), float(loss_scale), _ptr(loss), _ptr(lse), _ptr(logp),
                                            _ptr(ratio), _ptr(coef), _ptr(row_loss), _ptr(ws), _nbytes(ws),
                                            _stream(stream))
    _check(rc, "ps_lmhead_ppo_fwd_from_stats")


def ps_lmhead_ppo_bwd_vocab_shard(N, d, Vs, v0, V, dtype, Hpk, W_shard, tok, lse, coef, dH, dW_shard, flags, ws,
                                  stream=None):
    rc = lib().ps_lmhead_ppo_bwd_vocab_shard(N, d, Vs, v0, V, dtype, _ptr(Hpk), _ptr(W_shard), _ptr(tok), _ptr(lse),
                                             _ptr(coef), _ptr(dH), _ptr(dW_shard), flags, _ptr(ws), _nbytes(ws),
                                             _stream(stream))
    _check(rc, "ps_lmhead_ppo_bwd_vocab_shard")


def ps_lmhead_logit_store_size(N: int, V: int) -> int:
    return lib().ps_lmhead_logit_store_size(N, V)


def ps_lmhead_ppo_fwd_store(N, d, V, dtype, Hpk, W, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp, ratio,
                            coef, row_loss, store, ws, stream=None):
    rc = lib().ps_lmhead_ppo_fwd_store(N, d, V, dtype, _ptr(Hpk), _ptr(W), _ptr(tok), _ptr(oldlogp), _ptr(adv),
                                       _ptr(w), float(eps), float(loss_scale), _ptr(loss), _ptr(lse), _ptr(logp),
                                       _ptr(ratio), _ptr(coef), _ptr(row_loss), _ptr(store), _nbytes(store),
                                       _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_ppo_fwd_store")


def ps_lmhead_ppo_bwd_from_store_workspace_size() -> int:
    return lib().ps_lmhead_ppo_bwd_from_store_workspace_size()


def ps_lmhead_ppo_bwd_from_store(N, d, V, dtype, Hpk, W, tok, lse, logp, coef, store, dH, dW, flags, ws, stream=None):
    rc = lib().ps_lmhead_ppo_bwd_from_store(N, d, V, dtype, _ptr(Hpk), _ptr(W), _ptr(tok), _ptr(lse), _ptr(logp),
                                            _ptr(coef), _ptr(store), _nbytes(store), _ptr(dH), _ptr(dW), flags,
                                            _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_ppo_bwd_from_store")


def ps_lmhead_logit_stats_store(N, d, Vs, v0, dtype, Hpk, W_shard, tok, stats, ztok, store, ws, stream=None):
    rc = lib().ps_lmhead_logit_stats_store(N, d, Vs, v0, dtype, _ptr(Hpk), _ptr(W_shard), _ptr(tok), _ptr(stats),
                                           _ptr(ztok), _ptr(store), _nbytes(store), _ptr(ws), _nbytes(ws),
                                           _stream(stream))
    _check(rc, "ps_lmhead_logit_stats_store")


def ps_lmhead_ppo_bwd_vocab_shard_from_store(N, d, Vs, v0, V, dtype, Hpk, W_shard, tok, lse, logp, coef, store, dH,
                                             dW_shard, flags, ws, stream=None):
    rc = lib().ps_lmhead_ppo_bwd_vocab_shard_from_store(N, d, Vs, v0, V, dtype, _ptr(Hpk), _ptr(W_shard), _ptr(tok),
                                                        _ptr(lse), _ptr(logp), _ptr(coef), _ptr(store),
                                                        _nbytes(store), _ptr(dH), _ptr(dW_shard), flags, _ptr(ws),
                                                        _nbytes(ws), _stream(stream))
    _check(rc, "ps_lmhead_ppo_bwd_vocab_shard_from_store")


def ps_diag_gemm_bf16(M, N, K, a_mn_major, b_mn_major, A, lda, B, ldb, C, ldc, accumulate, ws, variant=0,
                      stream=None):
    rc = lib().ps_diag_gemm_bf16(M, N, K, int(a_mn_major), int(b_mn_major), _ptr(A), lda, _ptr(B), ldb, _ptr(C), ldc,
                                 int(accumulate), int(variant), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_diag_gemm_bf16")


def ps_diag_wait_timeout(timeout_ns, ws, stream=None):
    rc = lib().ps_diag_wait_timeout(int(timeout_ns), _ptr(ws), _nbytes(ws), _stream(stream))
    _check(rc, "ps_diag_wait_timeout")
