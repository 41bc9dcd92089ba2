"""Split key axis (partial softmax per key range, merged afterwards) vs the fp64 oracle."""
import numpy as np
import pytest

from gpu_helpers import assert_close, to_device

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


CASES = [
    ((1, 2, 256, 1000, 64, 64), 3),
    ((2, 1, 130, 4096, 128, 128), 4),
    ((1, 1, 5, 300, 128, 64), 2),
    ((1, 4, 64, 2500, 64, 128), 7),
    ((1, 1, 200, 128, 64, 64), 4),       # one key block: no split happens
    ((1, 8, 16, 8192, 128, 128), 16),    # decode-like: few query rows, long keys
]


@pytest.mark.parametrize("shape,splits", CASES, ids=lambda c: str(c))
def test_splitkv_parity(oracle, shape, splits):
    x = I.make_inputs(I.custom_config(*shape, dtype="bf16", seed=sum(shape) + splits))
    q, k, v = to_device(x)
    o = pkg.attn_fwd_splitkv(q, k, v, splits)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    assert_close(o.float().cpu().numpy(), oracle.attn(x.q, x.k, x.v, x.scale), "bf16",
                 f"{shape} splits={splits}")
    whole = pkg.attn_fwd(q, k, v).float()
    assert torch.max(torch.abs(whole - o.float())).item() <= 2e-2 * torch.max(torch.abs(whole)).item()


def test_splitkv_stress_with_plants(oracle):
    """Scores with sigma ~64 and planted dominant keys: the split maxima differ by hundreds."""
    cfg = I.custom_config(1, 2, 128, 2048, 128, 128, dtype="bf16", seed=55, q_sigma=8.0,
                          k_sigma=8.0, plants_per_head=4)
    x = I.make_inputs(cfg)
    q, k, v = to_device(x)
    o = pkg.attn_fwd_splitkv(q, k, v, 5)
    assert_close(o.float().cpu().numpy(), oracle.attn(x.q, x.k, x.v, x.scale), "bf16", "stress")
    of = o.float().cpu().numpy()
    for (b, h, i, kk) in x.plants:
        assert np.max(np.abs(of[b, h, i] - x.v[b, h, kk])) <= 1e-2 * max(1.0, np.max(np.abs(x.v[b, h, kk])))


def test_splitkv_rejects_small_workspace():
    x = I.make_inputs(I.custom_config(1, 1, 128, 1024, 64, 64, dtype="bf16", seed=3))
    q, k, v = to_device(x)
    need = pkg.moa_attn_splitkv_workspace_bytes(1, 1, 128, 1024, 64, 64, pkg.MOA_BF16, 4)
    ws = torch.empty(need - 16, dtype=torch.uint8, device=q.device)
    with pytest.raises(pkg.MoaError) as e:
        pkg.attn_fwd_splitkv(q, k, v, 4, workspace=ws)
    assert e.value.status == _lib.MOA_ERR_INVALID_ARG


def _sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def _auto_case(shape, seed):
    x = I.make_inputs(I.custom_config(*shape, dtype="bf16", seed=seed))
    q, k, v = to_device(x)
    rc, s, per, whole = pkg.moa_attn_split_plan(*shape[:4], pkg.MOA_SPLITS_AUTO, 0)
    assert rc == 0
    o = pkg.attn_fwd_splitkv(q, k, v, pkg.MOA_SPLITS_AUTO)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    return x, (q, k, v), o, (s, per, whole)


@pytest.mark.parametrize("shape", [(1, 4, 64, 4096, 128, 128), (2, 3, 300, 2000, 64, 64),
                                   (1, 5, 256, 3000, 128, 64)], ids=str)
def test_splitkv_auto_few_blocks(oracle, shape):
    """Fewer query blocks than SMs: every block's key axis is split (decode-like shapes, ragged
    query and key tails)."""
    x, (q, k, v), o, (s, per, whole) = _auto_case(shape, seed=sum(shape))
    assert s > 1 and whole == 0
    assert_close(o.float().cpu().numpy(), oracle.attn(x.q, x.k, x.v, x.scale), "bf16",
                 f"auto split {shape} splits={s}")
    need = pkg.moa_attn_splitkv_workspace_bytes(*shape, pkg.MOA_BF16, pkg.MOA_SPLITS_AUTO)
    assert need == s * shape[0] * shape[1] * shape[2] * (4 * shape[5] + 8)


def test_splitkv_auto_no_split_is_the_plain_kernel():
    """When the plan splits nothing the call is moa_attn_fwd: same bits."""
    S = _sms()
    shape = (1, S, 256, 640, 64, 64)
    x, (q, k, v), o, (s, per, whole) = _auto_case(shape, seed=5)
    assert s == 1
    assert torch.equal(o, pkg.attn_fwd(q, k, v))
    need = pkg.moa_attn_splitkv_workspace_bytes(*shape, pkg.MOA_BF16, pkg.MOA_SPLITS_AUTO)
    assert need == 0
