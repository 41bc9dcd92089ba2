"""Multi-rank host logic of bench.py on CPU: two gloo ranks (the path needs no collective on the
data; the timing reduction and the reference arm's rank-0-only rule are what N>1 adds)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # each rank reports its own (kernel ms, e2e ms); the job's time is the slowest rank's
    got = bench.reduce_max_over_ranks([10.0 + rank, 30.0 - rank])
    q.put((rank, got))
    dist.barrier()
    dist.destroy_process_group()


def test_timing_reduction_takes_slowest_rank():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = dict(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert results[0] == results[1] == [11.0, 30.0]


def test_whole_job_value_is_weak_scaling():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    one = bench.whole_job_tflops(1e12, 10, 1, 1000.0)
    two = bench.whole_job_tflops(1e12, 10, 2, 1000.0)
    assert one == pytest.approx(10.0) and two == pytest.approx(20.0)
    assert bench.reduce_max_over_ranks([1.5, 2.5]) == [1.5, 2.5]  # no process group: identity


def test_reference_arm_prints_on_rank_zero_only(monkeypatch, capsys):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    from paper_2606_07713_gb300 import inputs as I

    class A:
        steps, warmup = 1, 0
    monkeypatch.setenv("RANK", "1")
    bench.run_reference(A, I.CONFIGS[1])
    assert capsys.readouterr().out == ""
