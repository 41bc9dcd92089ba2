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
