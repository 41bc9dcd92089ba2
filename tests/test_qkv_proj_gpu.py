"""Fused input projections (moa_qkv_proj) vs the fp64 oracle, through the C ABI.

bf16 X and W enter the tensor-core products exactly and accumulate in fp32; the only rounding
that matters is the final one of each output to bf16 (relative 2^-9), plus fp32 summation
order over d_model terms.  Bound: |Q - Q_ref| <= 2^-8 |Q_ref| + d_model * 2^-23 * sum_c |X W|
element by element, checked as max|Q - Q_ref| / max|Q_ref| <= 1e-2 (BASELINE's bf16 bound is
2e-2), and exactness on small-integer inputs, where every product and sum is exact in fp32
and the bf16 result is exact.
"""
import numpy as np
import pytest

from gpu_helpers import rel_err

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


def bf16(a):
    bits = I.f32_to_bf16_bits(np.asarray(a, dtype=np.float32))
    return (I.bf16_bits_to_f32(bits),
            torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to("cuda:0"))


def run(xf, wf, H, dk, dv):
    x32, x = bf16(xf)
    w32, w = bf16(wf)
    q, k, v = pkg.qkv_proj(x, w, H, dk, dv)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    return x32, w32, tuple(t.float().cpu().numpy() for t in (q, k, v))


SHAPES = [  # B, N, d_model, H, d_k, d_v
    (1, 128, 64, 1, 64, 64),
    (2, 300, 256, 2, 64, 64),
    (1, 200, 520, 3, 128, 128),
    (3, 77, 128, 2, 128, 64),
    (2, 130, 96, 1, 64, 128),
    (1, 1, 8, 1, 64, 64),
    (2, 1000, 1024, 4, 64, 64),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_qkv_proj_parity(oracle, shape):
    B, N, d, H, dk, dv = shape
    r = np.random.default_rng(sum(shape))
    xf = r.normal(size=(B, N, d))
    wf = r.normal(size=(d, 2 * H * dk + H * dv)) / np.sqrt(d)
    x32, w32, got = run(xf, wf, H, dk, dv)
    ref = oracle.qkv_proj(x32, w32, H, dk, dv)
    for name, a, b in zip("QKV", got, ref):
        assert np.all(np.isfinite(a))
        err = rel_err(a, b)
        assert err <= 1e-2, f"{shape} {name}: {err:.3e}"


def test_qkv_proj_exact_on_small_integers(oracle):
    B, N, d, H, dk, dv = 2, 257, 192, 2, 64, 128
    r = np.random.default_rng(3)
    xf = r.integers(-2, 3, size=(B, N, d))
    wf = r.integers(-1, 2, size=(d, 2 * H * dk + H * dv))
    x32, w32, got = run(xf, wf, H, dk, dv)
    ref = oracle.qkv_proj(x32, w32, H, dk, dv)
    assert max(np.max(np.abs(t)) for t in ref) <= 256   # every value exact in bf16
    for a, b in zip(got, ref):
        assert np.array_equal(a.astype(np.float64), b)


def test_qkv_proj_feeds_attention(oracle):
    """Projection then attention (the step before the path, then the path) equals the oracle's
    attention of the oracle's projections, within the bf16 bound."""
    B, N, d, H, dk, dv = 1, 384, 256, 2, 64, 64
    r = np.random.default_rng(11)
    xf = r.normal(size=(B, N, d))
    wf = r.normal(size=(d, 2 * H * dk + H * dv)) / np.sqrt(d)
    x32, x = bf16(xf)
    w32, w = bf16(wf)
    q, k, v = pkg.qkv_proj(x, w, H, dk, dv)
    o = pkg.attn_fwd(q, k, v)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    qr, kr, vr = oracle.qkv_proj(x32, w32, H, dk, dv)
    # the oracle's attention on the bf16-rounded projections the kernel actually used
    qb, kb, vb = (t.float().cpu().numpy() for t in (q, k, v))
    for a, b in zip((qb, kb, vb), (qr, kr, vr)):
        assert rel_err(a, b) <= 1e-2
    ref = oracle.attn(qb, kb, vb, 1.0 / np.sqrt(dk))
    assert rel_err(o.float().cpu().numpy(), ref) <= 2e-2


@pytest.mark.parametrize("shape", [(1, 12800, 128, 2, 64, 64), (4, 2048, 256, 16, 64, 64)],
                         ids=["many-token-tiles", "bench-like"])
def test_qkv_proj_large_grids(oracle, shape):
    """Grids of several tiles per persistent CTA (both accumulators reused many times), checked
    on the first and the last 300 tokens of every batch entry (each token's outputs depend on
    that token's row of X only).  The last tokens come from the last, partly filled round of
    the persistent clusters (both CTAs of a cluster, second of a pair of token blocks)."""
    B, N, d, H, dk, dv = shape
    r = np.random.default_rng(sum(shape))
    xf = r.normal(size=(B, N, d))
    wf = r.normal(size=(d, 2 * H * dk + H * dv)) / np.sqrt(d)
    x32, w32, got = run(xf, wf, H, dk, dv)
    n = min(N, 300)
    for sl in (slice(0, n), slice(N - n, N)):
        ref = oracle.qkv_proj(np.ascontiguousarray(x32[:, sl]), w32, H, dk, dv)
        for name, a, b in zip("QKV", got, ref):
            err = rel_err(a[:, :, sl], b)
            assert err <= 1e-2, f"{shape} {name} tokens {sl}: {err:.3e}"
    for a in got:
        assert np.all(np.isfinite(a))


@pytest.mark.parametrize("shape", [(4, 2048, 1024, 16, 64, 64), (2, 8192, 4096, 32, 128, 128)],
                         ids=["bench-workload-2", "bench-workload-3"])
def test_qkv_proj_bench_shapes(oracle, shape):
    """The projections bench.py --pass qkv times (the cluster kernel, every pair item of the
    persistent grid), checked on the first and last 64 tokens of every batch entry."""
    B, N, d, H, dk, dv = shape
    r = np.random.default_rng(sum(shape))
    xf = r.normal(size=(B, N, d))
    wf = r.normal(size=(d, 2 * H * dk + H * dv)) / np.sqrt(d)
    x32, w32, got = run(xf, wf, H, dk, dv)
    for sl in (slice(0, 64), slice(N - 64, N)):
        ref = oracle.qkv_proj(np.ascontiguousarray(x32[:, sl]), w32, H, dk, dv)
        for name, a, b in zip("QKV", got, ref):
            err = rel_err(a[:, :, sl], b)
            assert err <= 1e-2, f"{shape} {name} tokens {sl}: {err:.3e}"
