"""The allocation-free split entry point (for callers that cannot allocate device memory).

It must give the same output as moa_attn_fwd_splitkv given a workspace of the caller's own,
call after call, although every call reuses the one scratch array inside the library.  This
file is named so that pytest collects it last; it also passes when run on its own.
"""
import ctypes

import numpy as np
import pytest

from paper_2606_07713_gb300 import _lib
from paper_2606_07713_gb300 import inputs as I


def test_noalloc_rejects_splits_larger_than_its_scratch():
    from paper_2606_07713_gb300 import build
    build.build()
    # 4 heads x 4096 query rows x 8 splits x (4*128 + 8) bytes = 68 MB > 16 MiB: refused before
    # any device work (the fake pointers below are never touched).
    rc = _lib.moa_attn_fwd_splitkv_noalloc(0x10000000, 0x20000000, 0x30000000, 0x40000000, 1, 4, 4096,
                                           4096, 128, 128, 0.08, _lib.MOA_BF16, 8, None)
    assert rc == _lib.MOA_ERR_UNSUPPORTED_SHAPE
    msg = _lib.moa_last_error()
    assert "scratch" in msg and str(_lib.MOA_NOALLOC_SCRATCH_BYTES) in msg


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from gpu_helpers import BF16_TOL, to_device
    _lib.lib()
    stream = torch.cuda.current_stream().cuda_stream
    # Two different problems back to back: the second call overwrites the scratch the first
    # one left behind, and must not be affected by it.
    cases = [((1, 8, 128, 8192, 128, 128), 8, 21), ((2, 4, 200, 3000, 64, 64), 5, 22)]
    for shape, splits, seed in cases:
        B, H, Nq, Nk, dk, dv = shape
        x = I.make_inputs(I.custom_config(*shape, dtype="bf16", seed=seed))
        q, k, v = to_device(x)
        scale = ctypes.c_float(x.scale).value
        o_ref = torch.empty((B, H, Nq, dv), dtype=torch.bfloat16, device=q.device)
        need = _lib.moa_attn_splitkv_workspace_bytes(B, H, Nq, Nk, dk, dv, _lib.MOA_BF16, splits)
        assert 0 < need <= _lib.MOA_NOALLOC_SCRATCH_BYTES
        ws = torch.empty(need, dtype=torch.uint8, device=q.device)
        rc = _lib.moa_attn_fwd_splitkv(q.data_ptr(), k.data_ptr(), v.data_ptr(), o_ref.data_ptr(),
                                       B, H, Nq, Nk, dk, dv, scale, _lib.MOA_BF16, splits,
                                       ws.data_ptr(), need, stream)
        assert rc == _lib.MOA_OK, _lib.moa_last_error()
        for call in range(2):
            o = torch.full((B, H, Nq, dv), float("nan"), dtype=torch.bfloat16, device=q.device)
            rc = _lib.moa_attn_fwd_splitkv_noalloc(q.data_ptr(), k.data_ptr(), v.data_ptr(),
                                                   o.data_ptr(), B, H, Nq, Nk, dk, dv, scale,
                                                   _lib.MOA_BF16, splits, stream)
            assert rc == _lib.MOA_OK, _lib.moa_last_error()
            torch.cuda.synchronize()
            # the same split and merge kernels on the same plan: the same bits, so a partial left
            # in the scratch by the previous call cannot hide inside a tolerance
            assert torch.equal(o, o_ref), (shape, call)
            got = o.float().cpu().numpy()
            want = o_ref.float().cpu().numpy()
            assert np.all(np.isfinite(got)), (shape, call)
            err = float(np.max(np.abs(got - want)) / np.max(np.abs(want)))
            assert err <= BF16_TOL, (shape, call, err)
    assert _lib.moa_get_device_status(stream) == _lib.MOA_OK


@pytest.mark.gpu
def test_noalloc_automatic_split_too_large_for_the_scratch_runs_unsplit():
    """With MOA_SPLITS_AUTO the library's own choice never fails for want of scratch: when the
    automatic plan's partials would not fit the static array, the call runs unsplit and gives
    moa_attn_fwd's bits."""
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from gpu_helpers import to_device
    _lib.lib()
    stream = torch.cuda.current_stream().cuda_stream
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # 64 heads x one 256-row query block = 64 blocks < the SM count: the automatic plan splits
    # every block's 16 key blocks in two, whose partials (2 x 16384 rows x 520 bytes, 17.0 MB)
    # exceed the 16 MiB array.
    shape = (1, 64, 256, 2048, 128, 128)
    B, H, Nq, Nk, dk, dv = shape
    rc, n_splits, _, _ = _lib.moa_attn_split_plan(B, H, Nq, Nk, _lib.MOA_SPLITS_AUTO, sms)
    assert rc == _lib.MOA_OK and n_splits > 1
    need = n_splits * B * H * Nq * (4 * dv + 8)
    assert need > _lib.MOA_NOALLOC_SCRATCH_BYTES
    x = I.make_inputs(I.custom_config(*shape, dtype="bf16", seed=23))
    q, k, v = to_device(x)
    scale = ctypes.c_float(x.scale).value
    o_ref = torch.empty((B, H, Nq, dv), dtype=torch.bfloat16, device=q.device)
    rc = _lib.moa_attn_fwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), o_ref.data_ptr(), B, H, Nq,
                           Nk, dk, dv, scale, _lib.MOA_BF16, stream)
    assert rc == _lib.MOA_OK, _lib.moa_last_error()
    for call in range(2):
        o = torch.full_like(o_ref, float("nan"))
        rc = _lib.moa_attn_fwd_splitkv_noalloc(q.data_ptr(), k.data_ptr(), v.data_ptr(),
                                               o.data_ptr(), B, H, Nq, Nk, dk, dv, scale,
                                               _lib.MOA_BF16, _lib.MOA_SPLITS_AUTO, stream)
        assert rc == _lib.MOA_OK, _lib.moa_last_error()
        torch.cuda.synchronize()
        assert torch.equal(o, o_ref), call
    assert _lib.moa_get_device_status(stream) == _lib.MOA_OK
