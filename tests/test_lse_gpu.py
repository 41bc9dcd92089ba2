"""Per-row log-sum-exp output (moa_attn_fwd_lse) vs the fp64 oracle, through the C ABI.

LSE_i = ln sum_k exp(scale <q_i, k_k>).  The kernels form the scores in fp32 from exact bf16 (or
fp32) products, so a score can be off by about d_k * 2^-24 * scale * sum_j |q_ij k_kj|; the LSE is
a smooth maximum of the scores and inherits that absolute error, plus the relative error of the
exp2/log2 (bf16 path: MUFU, about 2^-22) and of the final multiply by ln 2.
"""
import numpy as np
import pytest

from gpu_helpers import assert_close, lse_bound, to_device

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


def run_lse(x, scale=None):
    q, k, v = to_device(x)
    o, lse = pkg.attn_fwd_lse(q, k, v, x.scale if scale is None else scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    return o.float().cpu().numpy(), lse.cpu().numpy().astype(np.float64)


SHAPES = [
    (1, 1, 128, 128, 64, 64, "bf16"),
    (2, 3, 200, 300, 128, 128, "bf16"),
    (1, 2, 300, 1000, 64, 128, "bf16"),
    (2, 2, 513, 777, 128, 64, "bf16"),
    (1, 1, 1, 1, 64, 64, "bf16"),
    (1, 1, 5, 2, 128, 64, "bf16"),
    (3, 1, 130, 4096, 128, 128, "bf16"),
    (1, 1, 128, 128, 64, 64, "fp32"),
    (2, 3, 33, 70, 16, 8, "fp32"),
    (1, 1, 64, 65, 60, 100, "fp32"),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_lse_parity(oracle, shape):
    *dims, dtype = shape
    x = I.make_inputs(I.custom_config(*dims, dtype=dtype, seed=sum(dims) + 5))
    o, lse = run_lse(x)
    o_ref, lse_ref = oracle.attn_lse(x.q, x.k, x.v, x.scale)
    assert_close(o, o_ref, dtype, str(shape))
    err = np.abs(lse - lse_ref)
    assert np.all(np.isfinite(lse))
    assert np.all(err <= lse_bound(x, lse_ref)), f"max LSE error {err.max():.3e}"


@pytest.mark.parametrize("scale", [0.0, -0.3, 2.0])
def test_lse_unusual_scales(oracle, scale):
    x = I.make_inputs(I.custom_config(1, 2, 150, 260, 64, 64, dtype="bf16", seed=91))
    o, lse = run_lse(x, scale)
    o_ref, lse_ref = oracle.attn_lse(x.q, x.k, x.v, scale)
    assert_close(o, o_ref, "bf16", f"scale {scale}")
    if scale == 0.0:  # every score is 0: LSE = ln N_k exactly up to the log2/ln2 rounding
        assert np.max(np.abs(lse - np.log(260.0))) <= 1e-5
    assert np.all(np.abs(lse - lse_ref) <= lse_bound(x, lse_ref, scale))


def test_lse_large_scores_with_planted_rows(oracle):
    """Scores of size ~100 (Q sigma 8, d_k 128) and rows whose query equals one key: the
    rescale path runs and exp(s - m) underflows for most keys; LSE must still match."""
    cfg = I.custom_config(1, 2, 384, 1500, 128, 128, dtype="bf16", seed=17, q_sigma=8.0,
                          plants_per_head=4)
    x = I.make_inputs(cfg)
    o, lse = run_lse(x)
    o_ref, lse_ref = oracle.attn_lse(x.q, x.k, x.v, x.scale)
    assert_close(o, o_ref, "bf16", "large scores")
    assert np.all(np.abs(lse - lse_ref) <= lse_bound(x, lse_ref))


def test_lse_matches_plain_output_and_merges_halves(oracle):
    """O from the LSE entry point equals moa_attn_fwd's bit for bit, and the LSEs of two key
    halves merge to the whole: LSE = ln(exp(LSE_a) + exp(LSE_b)), O = w_a O_a + w_b O_b."""
    x = I.make_inputs(I.custom_config(2, 2, 256, 1024, 64, 64, dtype="bf16", seed=23))
    q, k, v = to_device(x)
    o_plain = pkg.attn_fwd(q, k, v, x.scale)
    o, lse = pkg.attn_fwd_lse(q, k, v, x.scale)
    oa, la = pkg.attn_fwd_lse(q, k[:, :, :512].contiguous(), v[:, :, :512].contiguous(), x.scale)
    ob, lb = pkg.attn_fwd_lse(q, k[:, :, 512:].contiguous(), v[:, :, 512:].contiguous(), x.scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    assert torch.equal(o_plain, o)
    la, lb, lse = (t.double().cpu().numpy() for t in (la, lb, lse))
    top = np.maximum(la, lb)
    merged = top + np.log(np.exp(la - top) + np.exp(lb - top))
    assert np.max(np.abs(merged - lse)) <= 1e-5 * (1 + np.max(np.abs(lse)))
    wa = np.exp(la - merged)[..., None]
    wb = np.exp(lb - merged)[..., None]
    om = wa * oa.double().cpu().numpy() + wb * ob.double().cpu().numpy()
    assert_close(om, oracle.attn(x.q, x.k, x.v, x.scale), "bf16", "merged halves")
