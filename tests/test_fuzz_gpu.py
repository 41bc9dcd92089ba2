"""Seeded random shapes through every bf16 entry point, against the fp64 oracle: forward,
forward with the log-sum-exp, split key axis (the library's own count and a random one), and
both backward forms.  Sizes are small and ragged (1 to ~700 rows, any mix of head dimensions,
scales of either sign) so that the oracle takes seconds; the point is the combinations the
hand-picked cases do not reach."""
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


def shapes(n, seed):
    r = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        B, H = int(r.integers(1, 4)), int(r.integers(1, 4))
        Nq = int(r.choice([1, 2, 7, 127, 128, 129, 255, 256, 257, int(r.integers(1, 700))]))
        Nk = int(r.choice([1, 3, 64, 127, 128, 129, 300, 511, 512, int(r.integers(1, 900))]))
        dk, dv = int(r.choice([64, 128])), int(r.choice([64, 128]))
        scale = float(r.choice([-1.0, 1.0]) * r.uniform(0.02, 0.3))
        out.append((B, H, Nq, Nk, dk, dv, round(scale, 4)))
    return out


def seed_of(shape):
    B, H, Nq, Nk, dk, dv, _ = shape
    return (B * 131 + H * 17 + Nq * 7 + Nk * 3 + dk + dv) % 10000


def close(got, ref, what):
    assert np.all(np.isfinite(got)), f"{what}: non-finite"
    m = float(np.max(np.abs(ref)))
    if m == 0.0:
        assert float(np.max(np.abs(got))) <= 1e-3, what
        return
    err = rel_err(got, ref)
    assert err <= BF16_TOL, f"{what}: {err:.3e}"


@pytest.mark.parametrize("shape", shapes(14, 2024), ids=str)
def test_fuzz_forward(oracle, shape):
    B, H, Nq, Nk, dk, dv, scale = shape
    x = I.make_inputs(I.custom_config(B, H, Nq, Nk, dk, dv, dtype="bf16", seed=seed_of(shape)))
    q, k, v = to_device(x)
    o_ref, lse_ref = oracle.attn_lse(x.q, x.k, x.v, scale)
    o = pkg.attn_fwd(q, k, v, scale)
    o2, lse = pkg.attn_fwd_lse(q, k, v, scale)
    r = np.random.default_rng(Nq + Nk)
    splits = int(r.integers(1, 9))
    o3 = pkg.attn_fwd_splitkv(q, k, v, splits, scale)
    o4 = pkg.attn_fwd_splitkv(q, k, v, pkg.MOA_SPLITS_AUTO, scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    for name, t in (("fwd", o), ("fwd_lse", o2), (f"split{splits}", o3), ("split_auto", o4)):
        close(t.float().cpu().numpy(), o_ref, f"{shape} {name}")
    assert torch.equal(o, o2), "the LSE output changes O"
    bound = 4e-6 * (1 + np.abs(lse_ref)) + 4 * dk * 2.0 ** -24 * abs(scale) * np.max(
        np.abs(x.q)) * np.max(np.abs(x.k)) * dk
    assert np.all(np.abs(lse.double().cpu().numpy() - lse_ref) <= bound), f"{shape} lse"


@pytest.mark.parametrize("shape", shapes(10, 77), ids=str)
def test_fuzz_backward(oracle, shape):
    B, H, Nq, Nk, dk, dv, scale = shape
    cfg = I.custom_config(B, H, Nq, Nk, dk, dv, dtype="bf16", seed=seed_of(shape))
    x = I.make_inputs(cfg)
    g, gb = I.make_grad_output(cfg)
    q, k, v = to_device(x)
    do = torch.from_numpy(np.ascontiguousarray(gb).view(np.int16)).view(torch.bfloat16).cuda()
    o, lse = pkg.attn_fwd_lse(q, k, v, scale)
    refs = oracle.attn_bwd(x.q, x.k, x.v, g, scale)
    paths = [False] + ([True] if dk == 64 and dv == 64 else [])
    for fused in paths:
        got = pkg.attn_bwd(q, k, v, o, lse, do, scale, fused=fused)
        torch.cuda.synchronize()
        pkg.check(pkg.get_device_status())
        for name, t, r in zip(("dQ", "dK", "dV"), got, refs):
            close(t.float().cpu().numpy(), r, f"{shape} {'fused' if fused else 'split'} {name}")
