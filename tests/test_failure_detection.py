"""Failure detection without faulting a GPU: the kernels' bounded waits give up, record
MOA_ERR_DEVICE_TIMEOUT in the device status word, and leave the context usable."""
import pytest

import paper_2606_07713_gb300 as pkg
from paper_2606_07713_gb300 import _lib


def test_selftest_rejects_bad_limits_without_gpu():
    from paper_2606_07713_gb300 import build
    build.build()
    assert _lib.moa_selftest_wait_timeout(0, None) == _lib.MOA_ERR_INVALID_ARG
    assert _lib.moa_selftest_wait_timeout(2 * 10 ** 10, None) == _lib.MOA_ERR_INVALID_ARG


@pytest.mark.gpu
def test_wait_that_never_completes_times_out_and_context_survives():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import numpy as np
    from gpu_helpers import assert_close, to_device
    from paper_2606_07713_gb300 import inputs as I
    import oracle
    s = torch.cuda.current_stream()
    assert pkg.get_device_status() == _lib.MOA_OK
    pkg.check(_lib.moa_selftest_wait_timeout(50_000_000, s.cuda_stream))  # 50 ms
    assert pkg.get_device_status() == _lib.MOA_ERR_DEVICE_TIMEOUT
    assert pkg.get_device_status() == _lib.MOA_OK  # read-and-clear
    # the context still runs real work correctly
    x = I.make_inputs(I.custom_config(1, 2, 256, 300, 64, 64, dtype="bf16", seed=3))
    o = pkg.attn_fwd(*to_device(x)).float().cpu().numpy()
    assert pkg.get_device_status() == _lib.MOA_OK
    assert_close(o, oracle.get().attn(x.q, x.k, x.v, x.scale), "bf16", "after timeout")


@pytest.mark.gpu
def test_debug_sync_mode_runs_every_entry_point_synchronously():
    """MOA_DEBUG_SYNC=1 (read once per process): every entry point synchronises after its launch
    and checks the status words; a clean run of each still returns MOA_OK."""
    import os
    import subprocess
    import sys
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    code = (
        "import torch, paper_2606_07713_gb300 as p\n"
        "q = torch.randn(1, 2, 300, 64, device='cuda', dtype=torch.bfloat16)\n"
        "k = torch.randn(1, 2, 500, 64, device='cuda', dtype=torch.bfloat16)\n"
        "v = torch.randn_like(k)\n"
        "o, lse = p.attn_fwd_lse(q, k, v)\n"
        "p.attn_fwd_splitkv(q, k, v, 3)\n"
        "p.attn_bwd(q, k, v, o, lse, torch.randn_like(o))\n"
        "x = torch.randn(1, 300, 128, device='cuda', dtype=torch.bfloat16)\n"
        "w = torch.randn(128, 192, device='cuda', dtype=torch.bfloat16)\n"
        "p.qkv_proj(x, w, 1, 64, 64)\n"
        "print('ok', p.get_device_status())\n")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, MOA_DEBUG_SYNC="1", PYTHONPATH=root)
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "ok 0" in r.stdout
