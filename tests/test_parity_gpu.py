"""CUDA path vs the fp64 oracle, element by element, through the C ABI (needs a GPU)."""
import math

import numpy as np
import pytest

from gpu_helpers import assert_close, bf16_tensor_from_f32, lse_bound, rel_err, to_device

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


def run(x, scale=None):
    q, k, v = to_device(x)
    o = pkg.attn_fwd(q, k, v, x.scale if scale is None else scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    return o.float().cpu().numpy()


# Shapes spanning several Q and key tiles, ragged tails, single rows/keys, all d_k/d_v pairs.
BF16_SHAPES = [
    (1, 1, 128, 128, 64, 64),
    (1, 1, 256, 256, 128, 128),
    (2, 3, 200, 300, 128, 128),
    (1, 2, 300, 1000, 64, 64),
    (1, 1, 1, 1, 64, 64),
    (1, 1, 5, 2, 128, 64),
    (1, 2, 300, 1000, 64, 128),
    (2, 2, 513, 777, 128, 64),
    (1, 1, 1000, 129, 64, 64),
    (3, 1, 130, 4096, 128, 128),
]


@pytest.mark.parametrize("shape", BF16_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_bf16_parity_full(oracle, shape):
    cfg = I.custom_config(*shape, dtype="bf16", seed=sum(shape))
    x = I.make_inputs(cfg)
    o = run(x)
    assert_close(o, oracle.attn(x.q, x.k, x.v, x.scale), "bf16", str(shape))


FP32_SHAPES = [
    (1, 1, 128, 128, 64, 64),
    (2, 3, 33, 70, 16, 8),
    (1, 2, 100, 257, 128, 128),
    (1, 1, 1, 1, 4, 4),
    (1, 1, 64, 65, 60, 100),
    (4, 4, 5, 1000, 32, 96),   # rows of a CTA past N_q; 16 key chunks through the double buffer
]


@pytest.mark.parametrize("shape", FP32_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_fp32_parity_full(oracle, shape):
    cfg = I.custom_config(*shape, dtype="fp32", seed=sum(shape))
    x = I.make_inputs(cfg)
    o = run(x)
    assert_close(o, oracle.attn(x.q, x.k, x.v, x.scale), "fp32", str(shape))


def test_workload_1_fp32_full(oracle):
    x = I.make_inputs(1)
    o = run(x)
    assert_close(o, oracle.attn(x.q, x.k, x.v, x.scale), "fp32", "workload 1")


@pytest.mark.parametrize("scale", [0.0, -0.3, 2.0])
def test_bf16_unusual_scales(oracle, scale):
    cfg = I.custom_config(1, 2, 150, 260, 64, 64, dtype="bf16", seed=77)
    x = I.make_inputs(cfg)
    o = run(x, scale)
    assert_close(o, oracle.attn(x.q, x.k, x.v, scale), "bf16", f"scale={scale}")


@pytest.mark.parametrize("dk,dv", [(64, 64), (128, 64)])
def test_bf16_grid_beyond_one_wave(oracle, dk, dv):
    """More 256-row work items than SMs (a second, nearly empty wave).  Every row of every head
    is checked, including rows of a half-valid second tile (N_q = 200) and the LSE output."""
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    H = n_sm + 10                       # n_sm + 10 work items
    cfg = I.custom_config(1, H, 200, 300, dk, dv, dtype="bf16", seed=H + dk)
    x = I.make_inputs(cfg)
    q, k, v = to_device(x)
    o, lse = pkg.attn_fwd_lse(q, k, v, x.scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    ref, lref = oracle.attn_lse(x.q, x.k, x.v, x.scale)
    assert_close(o.float().cpu().numpy(), ref, "bf16", f"tail d_k={dk} d_v={dv}")
    assert np.all(np.abs(lse.double().cpu().numpy() - lref) <= lse_bound(x, lref))


def test_fp32_tiled_kernel_on_a_large_grid(oracle):
    """fp32 problems with at least two 32-row CTAs per SM take the tiled kernel (smaller ones take
    the 8-row small kernel); every row checked."""
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    nq = 32 * ((2 * n_sm + 15) // 16)   # 16 heads x nq/32 CTAs >= 2 per SM
    cfg = I.custom_config(2, 8, nq, 300, 64, 64, dtype="fp32", seed=41)
    x = I.make_inputs(cfg)
    o = run(x)
    assert_close(o, oracle.attn(x.q, x.k, x.v, x.scale), "fp32", "tiled fp32 kernel")
