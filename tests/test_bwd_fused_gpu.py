"""Fused backward (moa_attn_bwd_fused: dK, dV and dQ from one tile kernel, d_k = d_v = 64) vs
the fp64 oracle, element by element, through the C ABI; and against the three-kernel
backward, which computes the same gradients with two extra tile products.

Tolerance: that of the three-kernel backward, max|g - g_ref| <= 2e-2 * max|g_ref|.  The fused
kernel rounds the same quantities to bf16 (W and dS before the products); dQ's fp32 sums of the
key blocks' products differ from one CTA's sum only in the order of fp32 additions.
"""
import numpy as np
import pytest

from gpu_helpers import BF16_TOL, rel_err, to_device

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import _lib  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


def bf16_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to("cuda:0")


def grads(x, g_bits, fused, scale=None):
    scale = x.scale if scale is None else scale
    q, k, v = to_device(x)
    do = bf16_dev(g_bits)
    o, lse = pkg.attn_fwd_lse(q, k, v, scale)
    out = pkg.attn_bwd(q, k, v, o, lse, do, scale, fused=fused)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    return out


SHAPES = [
    (1, 1, 128, 128, 64, 64),
    (1, 2, 300, 1000, 64, 64),
    (2, 3, 200, 300, 64, 64),
    (1, 1, 1000, 129, 64, 64),
    (2, 1, 513, 2048, 64, 64),
    (1, 1, 5, 3, 64, 64),
    (1, 1, 1, 1, 64, 64),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_fused_bwd_parity(oracle, shape):
    cfg = I.custom_config(*shape, dtype="bf16", seed=sum(shape) + 29)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    got = [t.float().cpu().numpy() for t in grads(x, gb, True)]
    ref = oracle.attn_bwd(x.q, x.k, x.v, g, x.scale)
    for name, a, b in zip(("dQ", "dK", "dV"), got, ref):
        assert np.all(np.isfinite(a)), f"{shape} {name}: non-finite"
        if np.max(np.abs(b)) == 0.0:
            assert np.max(np.abs(a)) <= 1e-3, f"{shape} {name}"
            continue
        err = rel_err(a, b)
        assert err <= BF16_TOL, f"{shape} {name}: max|g-g_ref|/max|g_ref| = {err:.3e}"


@pytest.mark.parametrize("scale", [-0.3, 2.0 / 8, 0.0])
def test_fused_bwd_other_scales(oracle, scale):
    """A negative scale (the maximum of the scaled scores is then at the smallest dot product),
    a larger one, and zero (uniform weights: dQ = dK = 0, dV = the column mean of dO)."""
    cfg = I.custom_config(1, 2, 260, 700, 64, 64, dtype="bf16", seed=77)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    got = [t.float().cpu().numpy() for t in grads(x, gb, True, scale=scale)]
    ref = oracle.attn_bwd(x.q, x.k, x.v, g, scale)
    for name, a, b in zip(("dQ", "dK", "dV"), got, ref):
        assert np.all(np.isfinite(a)), f"scale {scale} {name}"
        if np.max(np.abs(b)) == 0.0:
            assert np.max(np.abs(a)) <= 1e-3, f"scale {scale} {name}: {np.max(np.abs(a)):.3e} for 0"
            continue
        err = rel_err(a, b)
        assert err <= BF16_TOL, f"scale {scale} {name}: {err:.3e}"


def test_fused_matches_three_kernel_backward():
    """dK and dV: the same products in the same order of accumulation inside each CTA, so the
    same bits; dQ: the same products summed in another order (fp32), within bf16 rounding."""
    cfg = I.custom_config(2, 4, 700, 1500, 64, 64, dtype="bf16", seed=91)
    x = I.make_inputs(cfg)
    _, gb = I.make_grad_output(cfg)
    f = grads(x, gb, True)
    s = grads(x, gb, False)
    assert torch.equal(f[2], s[2]), "dV"
    assert torch.equal(f[1], s[1]), "dK"
    dq_err = (f[0].float() - s[0].float()).abs().max().item()
    assert dq_err <= 1e-2 * s[0].float().abs().max().item(), dq_err


def test_fused_dk_dv_reproducible():
    cfg = I.custom_config(1, 8, 1024, 1024, 64, 64, dtype="bf16", seed=5)
    x = I.make_inputs(cfg)
    _, gb = I.make_grad_output(cfg)
    a = grads(x, gb, True)
    b = grads(x, gb, True)
    assert torch.equal(a[1], b[1]) and torch.equal(a[2], b[2])
    # dQ: same values up to the order of fp32 additions
    assert (a[0].float() - b[0].float()).abs().max().item() <= 1e-2 * a[0].float().abs().max().item()


def test_fused_sum_rules():
    """The key gradients of a head sum to zero (the weights of a row sum to one) and the value
    gradients to the column sums of dO; dQ is orthogonal-free but <dQ, Q> = <dK, K>."""
    cfg = I.custom_config(1, 2, 256, 640, 64, 64, dtype="bf16", seed=17)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    dq, dk, dv = (t.double().cpu().numpy() for t in grads(x, gb, True))
    scale_dk = np.max(np.abs(dk))
    assert np.max(np.abs(dk.sum(axis=2))) <= 0.05 * scale_dk * np.sqrt(640)
    colsum = g.astype(np.float64).sum(axis=2)
    assert np.max(np.abs(dv.sum(axis=2) - colsum)) <= 2e-2 * np.max(np.abs(colsum)) + 1e-2
    lhs = np.sum(dq * x.q.astype(np.float64), axis=(2, 3))
    rhs = np.sum(dk * x.k.astype(np.float64), axis=(2, 3))
    assert np.max(np.abs(lhs - rhs)) <= 3e-2 * np.max(np.abs(rhs)) + 1e-2


def test_fused_rejects_other_shapes_and_dtypes():
    x = I.make_inputs(I.custom_config(1, 1, 128, 128, 128, 128, dtype="bf16", seed=3))
    _, gb = I.make_grad_output(x.cfg)
    q, k, v = to_device(x)
    o, lse = pkg.attn_fwd_lse(q, k, v, x.scale)
    with pytest.raises(pkg.MoaError) as e:
        pkg.attn_bwd(q, k, v, o, lse, bf16_dev(gb), x.scale, fused=True)
    assert e.value.status == _lib.MOA_ERR_UNSUPPORTED_SHAPE


def test_fused_bench_workload_sampled_heads(oracle):
    """The fused backward on bench.py's default backward workload (bf16 B=4 H=16 N=2048 d=64,
    the launch configuration `bench.py --pass bwd` times): three whole (b, h) slices, the last
    one from the last CTAs of the grid, element by element against the oracle."""
    cfg = I.CONFIGS[2]
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    dq, dk, dv = (t.float().cpu().numpy() for t in grads(x, gb, True))
    for (b, h) in [(0, 0), (2, 7), (3, 15)]:
        ref = oracle.attn_bwd(x.q[b:b + 1, h:h + 1], x.k[b:b + 1, h:h + 1], x.v[b:b + 1, h:h + 1],
                              g[b:b + 1, h:h + 1], x.scale)
        for name, a, r in zip(("dQ", "dK", "dV"), (dq, dk, dv), ref):
            err = rel_err(a[b:b + 1, h:h + 1], r)
            assert err <= BF16_TOL, f"workload 2 slice ({b},{h}) {name}: {err:.3e}"
