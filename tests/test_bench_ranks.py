"""The bench's multi-rank path on CPU: two gloo ranks, as torchrun would start
them for --gpus 2 (replicas of the repair, one per GPU).  The job's step time is
its slowest rank's, and its value counts every rank's rows over that time."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, step_ms, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(step_ms[rank], "cpu")
        q.put((rank, ms, bench.job_value(40, world, ms / 1e3)))
    finally:
        dist.destroy_process_group()


def test_two_ranks_report_the_slowest_rank_and_all_rows():
    torch = pytest.importorskip("torch")
    ctx = torch.multiprocessing.get_context("spawn")
    q = ctx.Queue()
    step_ms = [3.25, 3.5]
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, step_ms, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, value in got:
        assert ms == 3.5  # both ranks agree on the slowest step
        assert value == pytest.approx(2 * 40 / 3.5e-3)


def test_single_process_is_the_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(2.5, "cpu") == 2.5
    assert bench.job_value(40, 1, 2.5e-3) == pytest.approx(16000.0)
