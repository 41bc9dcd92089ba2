"""Closed-form and structural properties of the CUDA path, through the C ABI (needs a GPU)."""
import numpy as np
import pytest

from gpu_helpers import assert_close, bf16_tensor_from_f32, to_device

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


def inputs(shape, seed, dtype="bf16", **kw):
    return I.make_inputs(I.custom_config(*shape, dtype=dtype, seed=seed, **kw))


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_v_all_ones_gives_ones(dtype):
    x = inputs((1, 2, 300, 700, 128 if dtype == "bf16" else 64, 64), 5, dtype, q_sigma=3.0)
    q, k, _ = to_device(x)
    v = torch.ones((1, 2, 700, 64), dtype=q.dtype, device=q.device)
    o = pkg.attn_fwd(q, k, v).float().cpu().numpy()
    # bf16: P rounded to bf16 while l sums unrounded p (a few 2^-9 at most);
    # fp32: the BASELINE fp32 bound, 1e-5 of max|O_ref| = 1.
    tol = 2.0 ** -7 if dtype == "bf16" else 1e-5
    assert np.max(np.abs(o - 1.0)) <= tol


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_q_zero_gives_column_mean(dtype):
    x = inputs((2, 1, 260, 333, 64, 128 if dtype == "bf16" else 32), 6, dtype)
    _, k, v = to_device(x)
    q = torch.zeros((2, 1, 260, 64), dtype=k.dtype, device=k.device)
    o = pkg.attn_fwd(q, k, v).float().cpu().numpy()
    mean = x.v.astype(np.float64).mean(axis=2, keepdims=True)
    assert_close(o, np.broadcast_to(mean, o.shape), dtype, "Q=0")


def test_single_key_is_exact():
    x = inputs((2, 3, 257, 1, 128, 64), 7, q_sigma=5.0)
    q, k, v = to_device(x)
    o = pkg.attn_fwd(q, k, v)
    torch.cuda.synchronize()
    assert torch.equal(o, v.expand(2, 3, 257, 64))


def test_shift_invariance_through_inputs():
    """K[...,0] = 1 and Q[i,0] = delta_i add scale*delta_i to every score of row i."""
    x = inputs((1, 2, 200, 500, 64, 64), 8)
    qa = x.q.copy()
    ka = x.k.copy()
    ka[..., 0] = 1.0
    qa[..., 0] = 0.0
    qb = qa.copy()
    qb[..., 0] = np.random.default_rng(1).integers(-40, 40, size=qb.shape[:3]).astype(np.float32)
    k = bf16_tensor_from_f32(ka)
    v = to_device(x)[2]
    oa = pkg.attn_fwd(bf16_tensor_from_f32(qa), k, v).float().cpu().numpy()
    ob = pkg.attn_fwd(bf16_tensor_from_f32(qb), k, v).float().cpu().numpy()
    assert np.max(np.abs(oa - ob)) <= 2e-2 * np.max(np.abs(oa))


@pytest.mark.parametrize("dk,dv", [(128, 128), (64, 64), (128, 64)])
def test_heads_are_independent_bitwise(dk, dv):
    """A (b, h) slice alone gives the bits of the same slice in a batched call (d = 64 runs the
    one-tile kernel, the others the two-tile kernel)."""
    x = inputs((2, 3, 300, 400, dk, dv), 9)
    q, k, v = to_device(x)
    o = pkg.attn_fwd(q, k, v)
    for b, h in ((0, 0), (1, 2)):
        one = pkg.attn_fwd(q[b:b + 1, h:h + 1].contiguous(), k[b:b + 1, h:h + 1].contiguous(),
                           v[b:b + 1, h:h + 1].contiguous())
        assert torch.equal(one[0, 0], o[b, h])


@pytest.mark.parametrize("dk,dv,dtype", [(128, 128, "bf16"), (64, 64, "bf16"), (128, 64, "bf16"),
                                         (64, 64, "fp32")])
@pytest.mark.parametrize("world", [2, 3, 5])
def test_bh_ranges_reassemble_the_whole_call_bitwise(dk, dv, dtype, world):
    """The multi-GPU partition on one GPU: each rank's call runs on its contiguous block of
    (b, h) slices through pointer offsets into the same tensors (shard.block_view), writing its
    block of O in place; together the calls give the whole call's bits.  B*H = 14 is not a
    multiple of any of the rank counts."""
    from paper_2606_07713_gb300 import shard as SH
    x = inputs((2, 7, 300, 400, dk, dv), 19 + dk, dtype)
    q, k, v = to_device(x)
    whole = pkg.attn_fwd(q, k, v)
    parts = torch.full_like(whole, float("nan"))
    for lo, hi in SH.bh_ranges(14, world):
        pkg.attn_fwd(SH.block_view(q, lo, hi), SH.block_view(k, lo, hi), SH.block_view(v, lo, hi),
                     out=SH.block_view(parts, lo, hi))
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    assert torch.equal(parts, whole)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_run_to_run_bitwise_deterministic(dtype):
    x = inputs((2, 4, 1000, 1500, 64, 64), 10, dtype)
    q, k, v = to_device(x)
    a = pkg.attn_fwd(q, k, v)
    b = pkg.attn_fwd(q, k, v)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_output_guard_bands_untouched(dtype):
    """O is a window of a larger buffer filled with a sentinel: nothing outside it is written."""
    x = inputs((1, 2, 333, 250, 64, 64), 11, dtype)
    q, k, v = to_device(x)
    n = 1 * 2 * 333 * 64
    pad = 4096
    buf = torch.full((pad + n + pad,), -12345.0, dtype=q.dtype, device=q.device)
    o = buf[pad:pad + n].view(1, 2, 333, 64)
    pkg.attn_fwd(q, k, v, out=o)
    torch.cuda.synchronize()
    assert torch.all(buf[:pad] == -12345.0) and torch.all(buf[pad + n:] == -12345.0)
    assert not torch.any(o == -12345.0)


def test_staged_api_matches_device_api():
    x = inputs((2, 2, 400, 600, 128, 64), 12)
    q, k, v = to_device(x)
    o = pkg.attn_fwd(q, k, v)
    hq, hk, hv = (t.cpu().pin_memory() for t in (q, k, v))
    ho = torch.empty(o.shape, dtype=o.dtype).pin_memory()
    dq, dk, dv = (torch.empty_like(t) for t in (q, k, v))
    do = torch.empty_like(o)
    pkg.attn_fwd_staged(hq, hk, hv, ho, dq, dk, dv, do)
    torch.cuda.synchronize()
    assert torch.equal(ho, o.cpu())


@pytest.mark.parametrize("shape", [(4, 16, 4096, 4096, 64, 64), (1, 11, 8000, 16000, 128, 128)])
def test_staged_many_ranges_matches_device_api(shape):
    """Inputs of about 100 MB: six or seven head ranges of unequal size (the outer ones
    smallest), kernels alternating between two streams.  The host output must hold the bits of
    the device call's output for every head."""
    B, H, Nq, Nk, dk, dv = shape
    g = torch.Generator(device="cuda").manual_seed(61)
    q = torch.randn((B, H, Nq, dk), generator=g, device="cuda").to(torch.bfloat16)
    k = torch.randn((B, H, Nk, dk), generator=g, device="cuda").to(torch.bfloat16)
    v = torch.randn((B, H, Nk, dv), generator=g, device="cuda").to(torch.bfloat16)
    o = pkg.attn_fwd(q, k, v)
    hq, hk, hv = (t.cpu().pin_memory() for t in (q, k, v))
    ho = torch.full(o.shape, float("nan"), dtype=o.dtype).pin_memory()
    dq, dk_, dv_ = (torch.empty_like(t) for t in (q, k, v))
    do = torch.empty_like(o)
    pkg.attn_fwd_staged(hq, hk, hv, ho, dq, dk_, dv_, do)
    torch.cuda.synchronize()
    assert torch.equal(ho, o.cpu())


def test_device_status_clean_after_runs():
    x = inputs((1, 1, 128, 128, 64, 64), 13)
    pkg.attn_fwd(*to_device(x))
    assert pkg.get_device_status() == 0


def test_errors_reported_through_binding():
    x = inputs((1, 1, 64, 64, 64, 64), 14)
    q, k, v = to_device(x)
    with pytest.raises(pkg.MoaError) as e:
        pkg.attn_fwd(q, k, v, scale=float("nan"))
    assert e.value.status == 1
    q96 = torch.zeros((1, 1, 64, 96), dtype=torch.bfloat16, device=q.device)
    with pytest.raises(pkg.MoaError) as e:
        pkg.attn_fwd(q96, q96, v)
    assert e.value.status == 3


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_staged_pipeline_back_to_back_on_one_stream(dtype):
    """Two staged calls back to back on one user stream, sharing the device buffers: the second
    call's copies must wait for the first call's kernels, and synchronising that stream alone
    must make both host outputs valid.  9 heads: ranges of 3, 3, 3 (one range empty)."""
    shape = (3, 3, 200, 300, 64, 64)
    x1 = I.make_inputs(I.custom_config(*shape, dtype=dtype, seed=51))
    x2 = I.make_inputs(I.custom_config(*shape, dtype=dtype, seed=52))
    ref1 = pkg.attn_fwd(*to_device(x1)).cpu()
    ref2 = pkg.attn_fwd(*to_device(x2)).cpu()
    torch.cuda.synchronize()
    h1 = [t.cpu().pin_memory() for t in to_device(x1)]
    h2 = [t.cpu().pin_memory() for t in to_device(x2)]
    dq, dk, dv = (torch.empty_like(t) for t in to_device(x1))
    do = torch.empty(ref1.shape, dtype=ref1.dtype, device="cuda")
    ho1 = torch.empty(ref1.shape, dtype=ref1.dtype).pin_memory()
    ho2 = torch.empty(ref1.shape, dtype=ref1.dtype).pin_memory()
    s = torch.cuda.Stream()
    pkg.attn_fwd_staged(*h1, ho1, dq, dk, dv, do, stream=s)
    pkg.attn_fwd_staged(*h2, ho2, dq, dk, dv, do, stream=s)
    s.synchronize()
    assert torch.equal(ho1, ref1)
    assert torch.equal(ho2, ref2)
