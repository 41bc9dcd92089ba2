"""The B*H partition of a forward call across ranks (host logic; the multi-rank case runs as two
gloo processes on the CPU).  Each rank computes its range and its blocks of Q, K, V; the oracle
stands in for the forward on each block, and the blocks of O put back together must equal the
oracle's output for the whole call, bit for bit (each (b, h) slice is an independent problem)."""
import os
import socket

import numpy as np
import pytest

from paper_2606_07713_gb300 import inputs as I
from paper_2606_07713_gb300 import shard as SH

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("n", [0, 1, 2, 3, 7, 16, 64, 65, 1000])
@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
def test_ranges_cover_every_slice_once(n, world):
    rs = SH.bh_ranges(n, world)
    assert len(rs) == world
    owner = np.full(n, -1)
    for r, (lo, hi) in enumerate(rs):
        assert 0 <= lo <= hi <= n
        assert np.all(owner[lo:hi] == -1)
        owner[lo:hi] = r
    assert np.all(owner >= 0)
    sizes = [hi - lo for lo, hi in rs]
    assert max(sizes) - min(sizes) <= 1 and sizes == sorted(sizes, reverse=True)
    # contiguous, in rank order
    assert all(rs[r][1] == rs[r + 1][0] for r in range(world - 1))


def test_offsets_fall_on_slice_boundaries():
    B, H, N, d = 3, 5, 37, 24     # ragged: 15 slices over 4 ranks
    a = np.arange(B * H * N * d).reshape(B, H, N, d)
    flat = a.reshape(-1)
    for lo, hi in SH.bh_ranges(B * H, 4):
        off, cnt = SH.slice_offset(lo, N, d), SH.slice_numel(lo, hi, N, d)
        assert off % (N * d) == 0 and cnt % (N * d) == 0
        blk = SH.block(a, lo, hi)
        assert blk.shape == (1, hi - lo, N, d) and blk.flags.c_contiguous
        assert np.array_equal(blk.reshape(-1), flat[off:off + cnt])
        for j in range(hi - lo):
            b, h = divmod(lo + j, H)
            assert np.array_equal(blk[0, j], a[b, h])


def test_block_view_is_a_pointer_offset():
    torch = pytest.importorskip("torch")
    t = torch.arange(2 * 3 * 5 * 8, dtype=torch.float32).view(2, 3, 5, 8)
    for lo, hi in SH.bh_ranges(6, 4):
        v = SH.block_view(t, lo, hi)
        assert v.shape == (1, hi - lo, 5, 8) and v.is_contiguous()
        if hi > lo:
            assert v.data_ptr() == t.data_ptr() + 4 * SH.slice_offset(lo, 5, 8)
    with pytest.raises(ValueError):
        SH.block_view(t.transpose(2, 3), 0, 1)


def test_bad_partition_requests():
    for args in ((5, 0, 0), (5, 2, 2), (5, 2, -1), (-1, 2, 0)):
        with pytest.raises(ValueError):
            SH.bh_range(*args)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


CASE = (2, 3, 40, 70, 16, 8)   # B*H = 6 slices over 2 ranks; ragged sequence lengths


def _worker(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from paper_2606_07713_gb300 import inputs as In
    from paper_2606_07713_gb300 import shard as Sh
    cfg = In.custom_config(*CASE, dtype="fp32", seed=77)
    x = In.make_inputs(cfg)
    lo, hi = Sh.bh_range(cfg.shape.B * cfg.shape.H, world, rank)
    o_blk = oracle.get().attn(Sh.block(x.q, lo, hi), Sh.block(x.k, lo, hi),
                              Sh.block(x.v, lo, hi), x.scale)
    got = [None] * world
    dist.all_gather_object(got, (lo, hi, o_blk))
    if rank == 0:
        q.put(got)
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_reassemble_the_whole_call(oracle):
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    parts = q.get(timeout=180)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    cfg = I.custom_config(*CASE, dtype="fp32", seed=77)
    x = I.make_inputs(cfg)
    whole = oracle.attn(x.q, x.k, x.v, x.scale)
    s = cfg.shape
    assert [(lo, hi) for lo, hi, _ in parts] == SH.bh_ranges(s.B * s.H, world)
    joined = np.concatenate([o.reshape(-1, s.N_q, s.d_v) for _, _, o in parts])
    assert np.array_equal(joined.reshape(whole.shape), whole)
