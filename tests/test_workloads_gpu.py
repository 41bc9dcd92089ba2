"""The five workloads at full size, in the launch configuration bench.py times, against the
fp64 oracle: every row where the oracle finishes in seconds, else a seeded sample of at least 4096
rows that covers every (b, h), the first and last row of each head and every planted row (needs a
GPU)."""
import numpy as np
import pytest

from gpu_helpers import assert_close, sample_rows, to_device

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

import paper_2606_07713_gb300 as pkg  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pkg.lib()


@pytest.mark.parametrize("cid", [1, 2, 3, 4, 5])
def test_workload(oracle, cid):
    x = I.make_inputs(cid)
    s = x.shape
    q, k, v = to_device(x)
    o = pkg.attn_fwd(q, k, v, x.scale)
    torch.cuda.synchronize()
    pkg.check(pkg.get_device_status())
    full = cid in (1, 2, 4)
    if full:
        ref = oracle.attn(x.q, x.k, x.v, x.scale).reshape(-1, s.d_v)
        got = o.float().reshape(-1, s.d_v).cpu().numpy()
    else:
        rows = sample_rows(x)
        ref = oracle.rows(x.q, x.k, x.v, x.scale, rows)
        got = o.float().reshape(-1, s.d_v)[torch.from_numpy(rows).to(o.device)].cpu().numpy()
    err = assert_close(got, ref, x.cfg.dtype, f"workload {cid}")
    # also the relative RMS error and the worst row (reported; the bound above is the test)
    d = got.astype(np.float64) - ref
    rms = float(np.sqrt(np.mean(d * d)) / np.sqrt(np.mean(ref * ref)))
    worst = int(np.argmax(np.max(np.abs(d), axis=1)))
    wrow = worst if full else int(rows[worst])
    b, rem = divmod(wrow, s.H * s.N_q)
    h, i = divmod(rem, s.N_q)
    print(f"workload {cid}: max rel err {err:.2e}, rel RMS {rms:.2e}, worst row (b={b}, h={h}, i={i})")
    if x.plants:
        # One dominant key (margin > 30 in the scores, for every plant): the output row is that
        # key's value row.
        for (b, h, i, kk) in x.plants:
            sc = oracle.scores(x.q[b, h, i:i + 1], x.k[b, h], x.scale)[0]
            own = sc[kk]
            sc[kk] = -np.inf
            assert own - np.max(sc) > I.PLANT_MARGIN, (b, h, i, kk)
        of = o.float()
        for (b, h, i, kk) in x.plants:
            got_row = of[b, h, i].cpu().numpy()
            want = x.v[b, h, kk].astype(np.float64)
            assert np.max(np.abs(got_row - want)) <= 1e-2 * max(1.0, np.max(np.abs(want))), (b, h, i, kk)

