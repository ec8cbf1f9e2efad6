"""The benchmark's multi-rank host logic on two gloo ranks (CPU): every rank gets the slowest
rank's time, the whole-job value counts every rank's parameters, and the reference arm prints
from rank 0 only.  The outer step itself has no cross-GPU exchange (every rank runs its own
replica set), so this is all that differs at N > 1."""
import os
import socket

import pytest
import torch.multiprocessing as mp

from conftest import ROOT


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local_ms = 100.0 + 50.0 * rank
    total = bench.max_over_ranks(local_ms, dist, "cpu")
    dist.barrier()
    out[rank] = (total, bench.job_value(world, 1_000_000, 10, total))
    dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    assert res[0][0] == res[1][0] == 150.0
    # 2 ranks x 1e6 params x 10 steps in 0.15 s
    assert res[0][1] == pytest.approx(2 * 1_000_000 * 10 / 0.150)


def test_single_rank_keeps_its_time():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(42.0, None, "cpu") == 42.0
    assert bench.job_value(1, 100, 5, 1000.0) == 500.0


def test_reference_arm_prints_on_rank_0_only(monkeypatch, capsys):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")

    class Args:
        workload, steps, warmup, gpus = "llama_180m_k8", 1, 3, 2

    assert bench.run_reference(Args()) == 0
    assert capsys.readouterr().out == ""


def test_bench_report_helpers():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    table = [(0, 4, 4), (16, 3, 0), (19, 2, 8), (35, 4, 4)]
    assert bench.iters_by_shape(table, [7, 12, 9]) == {"4x4": {"7": 1, "9": 1}, "2x8": {"12": 1}}
    assert isinstance(bench.cpu_model(), str) and bench.cpu_model()
