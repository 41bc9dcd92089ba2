"""DNF attention forward for GB300 (sm_103a).

O = softmax(scale * Q K^T) V with a max-subtracted softmax, computed without any
score, probability or transposed-K array in device memory (the Denotational
Normal Form of Mullin & Hains, "Attention at the Theoretical Minimum").

The computation runs in libmoa_attn.so (hand-written CUDA: a tcgen05/TMEM/TMA
kernel for bf16 and a CUDA-core kernel for fp32).  This package is its thin
Python binding: PyTorch supplies device memory and the current stream, nothing
else.  There is no CPU fallback.
"""
from __future__ import annotations

import math

from ._lib import (MOA_BF16, MOA_FP32, MoaError, check, lib, moa_attn_dnf_bytes,  # noqa: F401
                   moa_attn_flops, moa_attn_fwd, moa_attn_fwd_staged, moa_attn_version,
                   moa_get_device_status, moa_last_error, moa_selftest_wait_timeout,
                   moa_attn_fwd_splitkv, moa_attn_splitkv_workspace_bytes, moa_attn_fwd_lse,
                   moa_attn_bwd, moa_attn_bwd_workspace_bytes, moa_qkv_proj,
                   moa_attn_split_plan, MOA_SPLITS_AUTO, moa_attn_bwd_fused,
                   moa_attn_bwd_fused_workspace_bytes)

__all__ = ["attn_fwd", "attn_fwd_staged", "get_device_status", "attn_flops", "dnf_bytes",
           "MOA_FP32", "MOA_BF16", "MoaError", "moa_attn_fwd", "moa_attn_fwd_staged",
           "moa_last_error", "moa_get_device_status", "moa_attn_flops", "moa_attn_dnf_bytes",
           "moa_attn_version", "moa_selftest_wait_timeout", "attn_fwd_splitkv",
           "moa_attn_fwd_splitkv", "moa_attn_splitkv_workspace_bytes", "attn_fwd_lse",
           "moa_attn_fwd_lse", "attn_bwd", "moa_attn_bwd", "moa_attn_bwd_workspace_bytes",
           "qkv_proj", "moa_qkv_proj", "moa_attn_split_plan", "MOA_SPLITS_AUTO",
           "moa_attn_bwd_fused", "moa_attn_bwd_fused_workspace_bytes"]


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return MOA_BF16
    if t.dtype == torch.float32:
        return MOA_FP32
    raise TypeError(f"unsupported dtype {t.dtype}; use torch.bfloat16 or torch.float32")


def _dims(q, k, v):
    if q.dim() != 4 or k.dim() != 4 or v.dim() != 4:
        raise ValueError("q, k, v must be [B, H, N, d]")
    B, H, Nq, dk = q.shape
    if tuple(k.shape[:2]) != (B, H) or tuple(v.shape[:2]) != (B, H):
        raise ValueError(f"batch/head mismatch: {tuple(q.shape)} {tuple(k.shape)} {tuple(v.shape)}")
    if k.shape[3] != dk or v.shape[2] != k.shape[2]:
        raise ValueError(f"shape mismatch: {tuple(q.shape)} {tuple(k.shape)} {tuple(v.shape)}")
    return B, H, Nq, k.shape[2], dk, v.shape[3]


def attn_fwd(q, k, v, scale: float | None = None, out=None, stream=None):
    """O = softmax(scale * q k^T) v for CUDA tensors [B, H, N, d] (bf16 or fp32).

    scale defaults to 1/sqrt(d_k).  Runs asynchronously on `stream` (default:
    torch's current stream of q's device) and returns `out` (allocated if None).
    """
    import torch
    for t in (q, k, v):
        if not t.is_cuda:
            raise ValueError("attn_fwd needs CUDA tensors")
        if not t.is_contiguous():
            raise ValueError("attn_fwd needs contiguous tensors")
    if not (q.dtype == k.dtype == v.dtype):
        raise TypeError("q, k, v must share one dtype")
    code = _dtype_code(q)
    B, H, Nq, Nk, dk, dv = _dims(q, k, v)
    if scale is None:
        scale = 1.0 / math.sqrt(dk)
    if out is None:
        out = torch.empty((B, H, Nq, dv), dtype=q.dtype, device=q.device)
    elif out.shape != (B, H, Nq, dv) or out.dtype != q.dtype or not out.is_contiguous():
        raise ValueError("out has the wrong shape, dtype or layout")
    with torch.cuda.device(q.device):
        s = stream if stream is not None else torch.cuda.current_stream(q.device)
        check(moa_attn_fwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), B, H, Nq, Nk,
                           dk, dv, float(scale), code, s.cuda_stream))
    return out


def attn_fwd_lse(q, k, v, scale: float | None = None, out=None, lse=None, stream=None):
    """(O, LSE): attn_fwd's output and the float32 [B, H, N_q] natural-log log-sum-exp of each
    row's scaled scores, ln sum_k exp(scale <q_i, k_k>)."""
    import torch
    for t in (q, k, v):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("attn_fwd_lse needs contiguous CUDA tensors")
    if not (q.dtype == k.dtype == v.dtype):
        raise TypeError("q, k, v must share one dtype")
    code = _dtype_code(q)
    B, H, Nq, Nk, dk, dv = _dims(q, k, v)
    if scale is None:
        scale = 1.0 / math.sqrt(dk)
    if out is None:
        out = torch.empty((B, H, Nq, dv), dtype=q.dtype, device=q.device)
    elif out.shape != (B, H, Nq, dv) or out.dtype != q.dtype or not out.is_contiguous():
        raise ValueError("out has the wrong shape, dtype or layout")
    if lse is None:
        lse = torch.empty((B, H, Nq), dtype=torch.float32, device=q.device)
    elif lse.shape != (B, H, Nq) or lse.dtype != torch.float32 or not lse.is_contiguous():
        raise ValueError("lse must be a contiguous float32 [B, H, N_q] tensor")
    with torch.cuda.device(q.device):
        s = stream if stream is not None else torch.cuda.current_stream(q.device)
        check(moa_attn_fwd_lse(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                               lse.data_ptr(), B, H, Nq, Nk, dk, dv, float(scale), code,
                               s.cuda_stream))
    return out, lse


def attn_bwd(q, k, v, o, lse, do, scale: float | None = None, workspace=None, stream=None,
             fused: bool = False):
    """(dQ, dK, dV) for O = softmax(scale q k^T) v given dO = dL/dO, from the forward's o and lse
    (attn_fwd_lse).  CUDA tensors [B, H, N, d]; lse float32 [B, H, N_q].  fused=True runs
    moa_attn_bwd_fused (bf16, d_k = d_v = 64; the key blocks' dQ tiles are added in fp32 by TMA
    reductions, in a run-dependent order)."""
    import torch
    for t in (q, k, v, o, do, lse):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("attn_bwd needs contiguous CUDA tensors")
    if not (q.dtype == k.dtype == v.dtype == o.dtype == do.dtype):
        raise TypeError("q, k, v, o, do must share one dtype")
    code = _dtype_code(q)
    B, H, Nq, Nk, dk, dv = _dims(q, k, v)
    if tuple(o.shape) != (B, H, Nq, dv) or tuple(do.shape) != (B, H, Nq, dv):
        raise ValueError("o and do must be [B, H, N_q, d_v]")
    if tuple(lse.shape) != (B, H, Nq) or lse.dtype != torch.float32:
        raise ValueError("lse must be float32 [B, H, N_q]")
    if scale is None:
        scale = 1.0 / math.sqrt(dk)
    dq = torch.empty_like(q)
    dkk = torch.empty_like(k)
    dvv = torch.empty_like(v)
    wsb = moa_attn_bwd_fused_workspace_bytes if fused else moa_attn_bwd_workspace_bytes
    call = moa_attn_bwd_fused if fused else moa_attn_bwd
    need = wsb(B, H, Nq, Nk, dk, dv, code)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=q.device)
    with torch.cuda.device(q.device):
        s = stream if stream is not None else torch.cuda.current_stream(q.device)
        check(call(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(), do.data_ptr(),
                   lse.data_ptr(), dq.data_ptr(), dkk.data_ptr(), dvv.data_ptr(), B, H, Nq, Nk, dk,
                   dv, float(scale), code, workspace.data_ptr(), workspace.numel(),
                   s.cuda_stream))
    return dq, dkk, dvv


def qkv_proj(x, w, H: int, d_k: int, d_v: int, out=None, stream=None):
    """(Q, K, V) = (X W_Q, X W_K, X W_V) in head-major layout [B, H, N, d] from x [B, N, d_model]
    and w [d_model, 2*H*d_k + H*d_v] (W_Q | W_K | W_V), bf16 CUDA tensors."""
    import torch
    for t in (x, w):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("qkv_proj needs contiguous CUDA tensors")
    if x.dim() != 3 or w.dim() != 2:
        raise ValueError("x must be [B, N, d_model] and w [d_model, 2*H*d_k + H*d_v]")
    if x.dtype != w.dtype:
        raise TypeError("x and w must share one dtype")
    code = _dtype_code(x)
    B, N, d = x.shape
    if tuple(w.shape) != (d, 2 * H * d_k + H * d_v):
        raise ValueError(f"w must be {(d, 2 * H * d_k + H * d_v)}, got {tuple(w.shape)}")
    if out is None:
        out = (torch.empty((B, H, N, d_k), dtype=x.dtype, device=x.device),
               torch.empty((B, H, N, d_k), dtype=x.dtype, device=x.device),
               torch.empty((B, H, N, d_v), dtype=x.dtype, device=x.device))
    q, k, v = out
    with torch.cuda.device(x.device):
        s = stream if stream is not None else torch.cuda.current_stream(x.device)
        check(moa_qkv_proj(x.data_ptr(), w.data_ptr(), q.data_ptr(), k.data_ptr(), v.data_ptr(),
                           B, N, d, H, d_k, d_v, code, s.cuda_stream))
    return q, k, v


def attn_fwd_splitkv(q, k, v, num_splits: int = MOA_SPLITS_AUTO, scale: float | None = None,
                     out=None, workspace=None, stream=None):
    """attn_fwd with the key axis split into up to num_splits ranges merged at the end.  With
    MOA_SPLITS_AUTO (0) the library chooses from q's device: when the 256-row query blocks leave
    SMs idle, every block's key axis is split so that the CTAs fill the SMs (if its cost model
    predicts a saving); otherwise nothing is split and the result is attn_fwd's.  The workspace
    (a CUDA uint8 tensor of at least moa_attn_splitkv_workspace_bytes(...) bytes) is allocated
    here when not given."""
    import torch
    for t in (q, k, v):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("attn_fwd_splitkv needs contiguous CUDA tensors")
    if not (q.dtype == k.dtype == v.dtype):
        raise TypeError("q, k, v must share one dtype")
    code = _dtype_code(q)
    B, H, Nq, Nk, dk, dv = _dims(q, k, v)
    if scale is None:
        scale = 1.0 / math.sqrt(dk)
    if out is None:
        out = torch.empty((B, H, Nq, dv), dtype=q.dtype, device=q.device)
    with torch.cuda.device(q.device):
        need = moa_attn_splitkv_workspace_bytes(B, H, Nq, Nk, dk, dv, code, int(num_splits))
        if workspace is None:
            workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=q.device)
        s = stream if stream is not None else torch.cuda.current_stream(q.device)
        check(moa_attn_fwd_splitkv(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), B, H,
                                   Nq, Nk, dk, dv, float(scale), code, int(num_splits),
                                   workspace.data_ptr(), workspace.numel(), s.cuda_stream))
    return out


def attn_fwd_staged(hq, hk, hv, ho, dq, dk_, dv_, do, scale: float | None = None, stream=None):
    """Host tensors in, host tensor out: copies hq/hk/hv to the device buffers dq/dk_/dv_,
    runs the kernel into do and copies it back into ho, all on one stream.  The result is in
    ho after the stream is synchronised."""
    import torch
    code = _dtype_code(dq)
    B, H, Nq, Nk, dk, dv = _dims(dq, dk_, dv_)
    for h, d in ((hq, dq), (hk, dk_), (hv, dv_), (ho, do)):
        if h.is_cuda or not d.is_cuda or h.shape != d.shape or h.dtype != d.dtype:
            raise ValueError("staged call needs matching host and device tensors")
        if not (h.is_contiguous() and d.is_contiguous()):
            raise ValueError("staged call needs contiguous tensors")
    if scale is None:
        scale = 1.0 / math.sqrt(dk)
    with torch.cuda.device(dq.device):
        s = stream if stream is not None else torch.cuda.current_stream(dq.device)
        check(moa_attn_fwd_staged(hq.data_ptr(), hk.data_ptr(), hv.data_ptr(), ho.data_ptr(),
                                  dq.data_ptr(), dk_.data_ptr(), dv_.data_ptr(), do.data_ptr(),
                                  B, H, Nq, Nk, dk, dv, float(scale), code, s.cuda_stream))
    return ho


def get_device_status(stream=None) -> int:
    """Synchronises the stream and returns/clears the kernels' timeout status word."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return moa_get_device_status(s.cuda_stream)


def attn_flops(B, H, N_q, N_k, d_k, d_v) -> float:
    return moa_attn_flops(B, H, N_q, N_k, d_k, d_v)


def dnf_bytes(B, H, N_q, N_k, d_k, d_v, dtype: int) -> float:
    return moa_attn_dnf_bytes(B, H, N_q, N_k, d_k, d_v, dtype)
