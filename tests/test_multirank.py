"""The N > 1 path of bench.py on CPU: ranks are replicas (each runs its own
batch, no exchange on the data path); the job's step time is the max over
ranks, taken with the one collective, and the throughput counts every rank's
images.  Two gloo ranks on 127.0.0.1, started with spawn."""
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, ws, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        got_ws, got_rank, _ = bench.dist_env()
        ms, value = bench.job_throughput(1.0 + rank, got_ws, 32, dist, "cpu")  # rank r took (1 + r) ms
        dist.barrier()
        q.put((got_rank, got_ws, ms, value))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_report_the_slowest_rank_and_all_images():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, ws, ms, value in res:
        assert ws == 2
        assert ms == pytest.approx(2.0)  # the slower rank's time, on every rank
        assert value == pytest.approx(2 * 32 / 2.0e-3)  # 64 images in 2 ms
    assert [r[0] for r in res] == [0, 1]


def test_single_process_throughput_has_no_collective():
    import bench
    assert bench.job_throughput(0.5, 1, 32) == (0.5, pytest.approx(64000.0))


def test_reference_arm_runs_on_rank_zero_only(capsys):
    import types
    import bench
    args = types.SimpleNamespace(steps=1, warmup=0)
    assert bench.run_reference(args, 2, 1) is None  # rank 1: no work, no line
    assert capsys.readouterr().out == ""
