"""The N > 1 path of bench.py on CPU: two replica processes over gloo (the
GPU run uses NCCL with one process per GPU). Each replica runs the whole
workload (weak scaling, no data-path collective); the job's time is the
slowest rank's, and the throughput counts the units of every rank."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
mp = pytest.importorskip("torch.multiprocessing")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        my_ms = [12.5, 20.0][rank]  # rank 1 is the slow replica
        ms = bench.max_over_ranks(my_ms, dist, "cpu")
        out[rank] = (ms, bench.whole_job_rate(256, world, ms))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_replicas_take_the_slowest_rank_and_count_every_rank():
    world = 2
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    assert res[0] == res[1]
    ms, rate = res[0]
    assert ms == 20.0
    assert rate == pytest.approx(2 * 256 / 0.020)


def test_single_process_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(7.0, None, "cpu") == 7.0
    assert bench.whole_job_rate(100, 1, 50.0) == pytest.approx(2000.0)


def test_reference_arm_under_torchrun_prints_only_on_rank_zero(capsys):
    sys.path.insert(0, ROOT)
    import bench

    class A:
        workload, steps, warmup, gpus = "135m_b1_s16_n16", 1, 0, 2
    bench.run_reference(A, rank=1, world=2)
    assert capsys.readouterr().out == ""
