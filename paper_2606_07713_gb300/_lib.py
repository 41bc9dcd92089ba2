"""ctypes binding of libmoa_attn.so: the C ABI of include/moa_attn.h, name for name.

Argument marshalling only.  Every step of the attention computation runs in
the library's CUDA kernels; there is no Python or CPU fallback, and loading
fails loudly if the library has not been built.
"""
from __future__ import annotations

import ctypes
import os
import threading

MOA_FP32 = 0
MOA_BF16 = 1

MOA_OK = 0
MOA_ERR_INVALID_ARG = 1
MOA_ERR_UNSUPPORTED_DTYPE = 2
MOA_ERR_UNSUPPORTED_SHAPE = 3
MOA_ERR_MISALIGNED = 4
MOA_ERR_CUDA = 5
MOA_ERR_DEVICE_TIMEOUT = 6

STATUS_NAMES = {
    MOA_OK: "MOA_OK",
    MOA_ERR_INVALID_ARG: "MOA_ERR_INVALID_ARG",
    MOA_ERR_UNSUPPORTED_DTYPE: "MOA_ERR_UNSUPPORTED_DTYPE",
    MOA_ERR_UNSUPPORTED_SHAPE: "MOA_ERR_UNSUPPORTED_SHAPE",
    MOA_ERR_MISALIGNED: "MOA_ERR_MISALIGNED",
    MOA_ERR_CUDA: "MOA_ERR_CUDA",
    MOA_ERR_DEVICE_TIMEOUT: "MOA_ERR_DEVICE_TIMEOUT",
}

# Every function declared in include/moa_attn.h: name -> (restype, argtypes).
_VP = ctypes.c_void_p
_I64 = ctypes.c_int64
SIGNATURES = {
    "moa_attn_fwd": (ctypes.c_int, [_VP, _VP, _VP, _VP, _I64, _I64, _I64, _I64, _I64, _I64,
                                    ctypes.c_float, ctypes.c_int, _VP]),
    "moa_attn_fwd_lse": (ctypes.c_int, [_VP, _VP, _VP, _VP, _VP, _I64, _I64, _I64, _I64, _I64,
                                        _I64, ctypes.c_float, ctypes.c_int, _VP]),
    "moa_attn_bwd": (ctypes.c_int, [_VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _I64, _I64, _I64,
                                    _I64, _I64, _I64, ctypes.c_float, ctypes.c_int, _VP,
                                    ctypes.c_size_t, _VP]),
    "moa_attn_bwd_workspace_bytes": (ctypes.c_size_t, [_I64, _I64, _I64, _I64, _I64, _I64,
                                                       ctypes.c_int]),
    "moa_attn_bwd_fused": (ctypes.c_int, [_VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _I64, _I64,
                                          _I64, _I64, _I64, _I64, ctypes.c_float, ctypes.c_int,
                                          _VP, ctypes.c_size_t, _VP]),
    "moa_attn_bwd_fused_workspace_bytes": (ctypes.c_size_t, [_I64, _I64, _I64, _I64, _I64, _I64,
                                                             ctypes.c_int]),
    "moa_qkv_proj": (ctypes.c_int, [_VP, _VP, _VP, _VP, _VP, _I64, _I64, _I64, _I64, _I64, _I64,
                                    ctypes.c_int, _VP]),
    "moa_attn_fwd_staged": (ctypes.c_int, [_VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _I64, _I64,
                                           _I64, _I64, _I64, _I64, ctypes.c_float, ctypes.c_int,
                                           _VP]),
    "moa_attn_fwd_splitkv": (ctypes.c_int, [_VP, _VP, _VP, _VP, _I64, _I64, _I64, _I64, _I64,
                                            _I64, ctypes.c_float, ctypes.c_int, ctypes.c_int,
                                            _VP, ctypes.c_size_t, _VP]),
    "moa_attn_splitkv_workspace_bytes": (ctypes.c_size_t, [_I64, _I64, _I64, _I64, _I64, _I64,
                                                           ctypes.c_int, ctypes.c_int]),
    "moa_attn_fwd_splitkv_noalloc": (ctypes.c_int, [_VP, _VP, _VP, _VP, _I64, _I64, _I64, _I64,
                                                    _I64, _I64, ctypes.c_float, ctypes.c_int,
                                                    ctypes.c_int, _VP]),
    "moa_attn_split_plan": (ctypes.c_int, [_I64, _I64, _I64, _I64, ctypes.c_int, ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_int),
                                           ctypes.POINTER(ctypes.c_int),
                                           ctypes.POINTER(ctypes.c_int64)]),
    "moa_last_error": (ctypes.c_char_p, []),
    "moa_get_device_status": (ctypes.c_int, [_VP]),
    "moa_selftest_wait_timeout": (ctypes.c_int, [ctypes.c_uint64, _VP]),
    "moa_attn_flops": (ctypes.c_double, [_I64, _I64, _I64, _I64, _I64, _I64]),
    "moa_attn_dnf_bytes": (ctypes.c_double, [_I64, _I64, _I64, _I64, _I64, _I64, ctypes.c_int]),
    "moa_attn_version": (ctypes.c_int, []),
}

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build", "libmoa_attn.so")
_lib = None
_lock = threading.Lock()


class MoaError(RuntimeError):
    """A non-OK status from the library, with its moa_last_error() text."""

    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


def lib() -> ctypes.CDLL:
    """The loaded libmoa_attn.so.  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"{LIB_PATH} is missing: build it with "
                    "`python -c 'import __graft_entry__ as g; g.build()'` (needs nvcc)")
            L = ctypes.CDLL(LIB_PATH)
            for name, (res, args) in SIGNATURES.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def check(status: int) -> None:
    if status != MOA_OK:
        raise MoaError(status, (lib().moa_last_error() or b"").decode(errors="replace"))


# -- thin wrappers with the C names ----------------------------------------------------------
def moa_attn_fwd(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream) -> int:
    return lib().moa_attn_fwd(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream)


def moa_attn_fwd_lse(Q, K, V, O, LSE, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream) -> int:
    return lib().moa_attn_fwd_lse(Q, K, V, O, LSE, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream)


def moa_attn_bwd(Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                 workspace, workspace_bytes, stream) -> int:
    return lib().moa_attn_bwd(Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v, scale,
                              dtype, workspace, workspace_bytes, stream)


def moa_attn_bwd_workspace_bytes(B, H, N_q, N_k, d_k, d_v, dtype) -> int:
    return lib().moa_attn_bwd_workspace_bytes(B, H, N_q, N_k, d_k, d_v, dtype)


def moa_attn_bwd_fused(Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                       workspace, workspace_bytes, stream) -> int:
    return lib().moa_attn_bwd_fused(Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v,
                                    scale, dtype, workspace, workspace_bytes, stream)


def moa_attn_bwd_fused_workspace_bytes(B, H, N_q, N_k, d_k, d_v, dtype) -> int:
    return lib().moa_attn_bwd_fused_workspace_bytes(B, H, N_q, N_k, d_k, d_v, dtype)


def moa_qkv_proj(X, W, Q, K, V, B, N, d_model, H, d_k, d_v, dtype, stream) -> int:
    return lib().moa_qkv_proj(X, W, Q, K, V, B, N, d_model, H, d_k, d_v, dtype, stream)


def moa_attn_fwd_staged(hQ, hK, hV, hO, dQ, dK, dV, dO, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                        stream) -> int:
    return lib().moa_attn_fwd_staged(hQ, hK, hV, hO, dQ, dK, dV, dO, B, H, N_q, N_k, d_k, d_v,
                                     scale, dtype, stream)


def moa_attn_fwd_splitkv(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, num_splits,
                         workspace, workspace_bytes, stream) -> int:
    return lib().moa_attn_fwd_splitkv(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                                      num_splits, workspace, workspace_bytes, stream)


def moa_attn_splitkv_workspace_bytes(B, H, N_q, N_k, d_k, d_v, dtype, num_splits) -> int:
    return lib().moa_attn_splitkv_workspace_bytes(B, H, N_q, N_k, d_k, d_v, dtype, num_splits)


def moa_attn_fwd_splitkv_noalloc(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, num_splits,
                                 stream) -> int:
    return lib().moa_attn_fwd_splitkv_noalloc(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                                              num_splits, stream)


def moa_attn_split_plan(B, H, N_q, N_k, num_splits, sm_count) -> tuple[int, int, int, int]:
    """(status, splits, key_blocks_per_split, whole_query_blocks) of moa_attn_split_plan."""
    s, per = ctypes.c_int(0), ctypes.c_int(0)
    whole = ctypes.c_int64(0)
    rc = lib().moa_attn_split_plan(B, H, N_q, N_k, num_splits, sm_count, ctypes.byref(s),
                                   ctypes.byref(per), ctypes.byref(whole))
    return rc, s.value, per.value, whole.value


# MOA_NOALLOC_SCRATCH_BYTES and MOA_SPLITS_AUTO of include/moa_attn.h
MOA_NOALLOC_SCRATCH_BYTES = 16 << 20
MOA_SPLITS_AUTO = 0


def moa_last_error() -> str:
    return (lib().moa_last_error() or b"").decode(errors="replace")


def moa_get_device_status(stream) -> int:
    return lib().moa_get_device_status(stream)


def moa_selftest_wait_timeout(limit_ns, stream) -> int:
    return lib().moa_selftest_wait_timeout(limit_ns, stream)


def moa_attn_flops(B, H, N_q, N_k, d_k, d_v) -> float:
    return lib().moa_attn_flops(B, H, N_q, N_k, d_k, d_v)


def moa_attn_dnf_bytes(B, H, N_q, N_k, d_k, d_v, dtype) -> float:
    return lib().moa_attn_dnf_bytes(B, H, N_q, N_k, d_k, d_v, dtype)


def moa_attn_version() -> int:
    return lib().moa_attn_version()
