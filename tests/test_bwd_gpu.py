"""Backward pass (moa_attn_bwd) vs the fp64 oracle, element by element, through the C ABI.

The GPU path takes O and LSE from its own forward kernel (moa_attn_fwd_lse); the oracle
recomputes everything in fp64 from Q, K, V and dO.  Tolerance: the bf16 bound of the forward
tests, max|g - g_ref| <= 2e-2 * max|g_ref| per gradient.  A model of the bf16 roundings the
kernels make (O, the weights W and dS rounded to bf16 before the products) gives 1.4e-3 to
2.9e-3 on these shapes, so the bound has a margin of about 7.
"""
import numpy as np
import pytest

from gpu_helpers import BF16_TOL, rel_err, to_device

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


def bf16_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to("cuda:0")


def run_bwd(x, g_bits, scale=None, g32=None):
    scale = x.scale if scale is None else scale
    q, k, v = to_device(x)
    do = bf16_dev(g_bits) if g32 is None else torch.from_numpy(np.ascontiguousarray(g32)).to("cuda:0")
    o, lse = pkg.attn_fwd_lse(q, k, v, scale)
    dq, dk, dv = pkg.attn_bwd(q, k, v, o, lse, do, scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    return tuple(t.float().cpu().numpy() for t in (dq, dk, dv))


def check_grads(got, ref, what):
    for name, a, b in zip(("dQ", "dK", "dV"), got, ref):
        assert np.all(np.isfinite(a)), f"{what} {name}: non-finite"
        if np.max(np.abs(b)) == 0.0:
            # an exactly zero gradient (one key): only the rounding of dP - D remains
            assert np.max(np.abs(a)) <= 1e-3, f"{what} {name}: {np.max(np.abs(a)):.3e} for 0"
            continue
        err = rel_err(a, b)
        assert err <= BF16_TOL, f"{what} {name}: max|g-g_ref|/max|g_ref| = {err:.3e}"


SHAPES = [
    (1, 1, 128, 128, 64, 64),
    (1, 1, 256, 256, 128, 128),
    (2, 3, 200, 300, 128, 128),
    (1, 2, 300, 1000, 64, 64),
    (1, 2, 300, 1000, 64, 128),
    (2, 2, 513, 777, 128, 64),
    (1, 1, 1000, 129, 64, 64),
    (3, 1, 130, 2048, 128, 128),
    (1, 1, 5, 3, 64, 64),
    (1, 1, 1, 1, 128, 128),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_bwd_parity(oracle, shape):
    cfg = I.custom_config(*shape, dtype="bf16", seed=sum(shape) + 11)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    got = run_bwd(x, gb)
    ref = oracle.attn_bwd(x.q, x.k, x.v, g, x.scale)
    check_grads(got, ref, str(shape))


@pytest.mark.parametrize("scale", [-0.3, 2.0 / 8])
def test_bwd_other_scales(oracle, scale):
    cfg = I.custom_config(1, 2, 150, 260, 64, 64, dtype="bf16", seed=93)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    got = run_bwd(x, gb, scale)
    check_grads(got, oracle.attn_bwd(x.q, x.k, x.v, g, scale), f"scale {scale}")


def test_bwd_large_scores_and_planted_rows(oracle):
    cfg = I.custom_config(1, 2, 384, 700, 128, 128, dtype="bf16", seed=19, q_sigma=4.0,
                          plants_per_head=4)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    check_grads(run_bwd(x, gb), oracle.attn_bwd(x.q, x.k, x.v, g, x.scale), "large scores")


def test_bwd_single_key_closed_form():
    """One key: the weights are all 1, so dQ = dK = 0 up to the rounding of dP - D, and
    dV = sum over the query rows of dO."""
    cfg = I.custom_config(1, 2, 300, 1, 64, 64, dtype="bf16", seed=7)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    dq, dk, dv = run_bwd(x, gb)
    assert np.max(np.abs(dq)) <= 1e-2 and np.max(np.abs(dk)) <= 1e-1
    ref = g.astype(np.float64).sum(axis=2)
    assert rel_err(dv[:, :, 0], ref) <= 1e-2


def test_bwd_gradients_sum_rules():
    """Properties at a size the oracle would be slow on: each head's dK rows sum to ~0 and its
    dV rows to sum_i dO_i (weights sum to one per row)."""
    cfg = I.custom_config(1, 4, 2048, 2048, 64, 64, dtype="bf16", seed=29)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    dq, dk, dv = run_bwd(x, gb)
    gsum = g.astype(np.float64).sum(axis=2)
    assert rel_err(dv.astype(np.float64).sum(axis=2), gsum) <= 2e-2
    assert np.max(np.abs(dk.astype(np.float64).sum(axis=2))) <= 2e-2 * np.max(np.abs(dk)) * np.sqrt(2048)


FP32_SHAPES = [
    (1, 1, 128, 128, 64, 64),
    (2, 3, 33, 70, 16, 8),
    (1, 2, 100, 257, 128, 128),
    (1, 1, 64, 65, 60, 100),
    (1, 1, 1, 1, 4, 4),
]


@pytest.mark.parametrize("shape", FP32_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_bwd_fp32_parity(oracle, shape):
    """The fp32 CUDA-core backward: fp32 products and sums, expf for the weights, against the
    fp64 oracle within 2e-5 of max per gradient: the forward's O and LSE and the row sums D are
    fp32 (relative 2^-24 per operation, sums of up to a few hundred terms), and dP - D cancels,
    which is why the bound is twice the forward's 1e-5."""
    cfg = I.custom_config(*shape, dtype="fp32", seed=sum(shape) + 17)
    x = I.make_inputs(cfg)
    g, _ = I.make_grad_output(cfg)
    got = run_bwd(x, None, g32=g)
    ref = oracle.attn_bwd(x.q, x.k, x.v, g, x.scale)
    for name, a, b in zip(("dQ", "dK", "dV"), got, ref):
        assert np.all(np.isfinite(a)), f"{shape} {name}: non-finite"
        if np.max(np.abs(b)) == 0.0:
            assert np.max(np.abs(a)) <= 1e-6, f"{shape} {name}"
            continue
        err = rel_err(a, b)
        assert err <= 2e-5, f"{shape} {name}: {err:.3e}"


def test_bwd_bench_workload_sampled_heads(oracle):
    """The backward on `bench.py --pass bwd`'s default workload (bf16 B=4 H=16 N=2048 d=64, in the
    launch configuration it times), two whole (b, h) slices checked against the
    oracle element by element (each slice's gradients depend only on that slice)."""
    cfg = I.CONFIGS[2]
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    dq, dk, dv = run_bwd(x, gb)
    for (b, h) in [(0, 0), (3, 11)]:
        ref = oracle.attn_bwd(x.q[b:b + 1, h:h + 1], x.k[b:b + 1, h:h + 1], x.v[b:b + 1, h:h + 1],
                              g[b:b + 1, h:h + 1], x.scale)
        got = tuple(t[b:b + 1, h:h + 1] for t in (dq, dk, dv))
        check_grads(got, ref, f"workload 2 slice ({b},{h})")


def test_bwd_d128_workload_sampled_head(oracle):
    """The three-kernel backward on the d=128 workload bench.py --pass bwd --workload 3 times
    (bf16 B=2 H=32 N=8192), the last (b, h) slice against the oracle element by element."""
    cfg = I.CONFIGS[3]
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    dq, dk, dv = run_bwd(x, gb)
    b, h = 1, 31
    ref = oracle.attn_bwd(x.q[b:b + 1, h:h + 1], x.k[b:b + 1, h:h + 1], x.v[b:b + 1, h:h + 1],
                          g[b:b + 1, h:h + 1], x.scale)
    got = tuple(t[b:b + 1, h:h + 1] for t in (dq, dk, dv))
    check_grads(got, ref, f"workload 3 slice ({b},{h})")


@pytest.mark.parametrize("dtype,dk,dv", [("bf16", 64, 64), ("bf16", 128, 128), ("bf16", 128, 64),
                                         ("fp32", 64, 64)])
def test_three_kernel_backward_bitwise_reproducible(dtype, dk, dv):
    """moa_attn_bwd adds every gradient in a fixed order, so two calls on the same inputs give
    the same bits (the reproducible choice; moa_attn_bwd_fused's dQ is not)."""
    cfg = I.custom_config(2, 4, 700, 900, dk, dv, dtype=dtype, seed=dk + dv)
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    q, k, v = to_device(x)
    do = bf16_dev(gb) if dtype == "bf16" else torch.from_numpy(np.ascontiguousarray(g)).to("cuda:0")
    o, lse = pkg.attn_fwd_lse(q, k, v, x.scale)
    a = pkg.attn_bwd(q, k, v, o, lse, do, x.scale)
    b = pkg.attn_bwd(q, k, v, o, lse, do, x.scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    for name, ta, tb in zip(("dQ", "dK", "dV"), a, b):
        assert torch.equal(ta, tb), name
