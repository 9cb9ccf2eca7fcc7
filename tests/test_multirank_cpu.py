"""bench.py's multi-rank path on the CPU: world size 2 over gloo (one process per
rank, as torchrun launches them).  The timing reported is the slowest rank's,
every rank sees the same value, and the whole-job rate counts all ranks' tokens
over that time.  No GPU: the GPU ranks run the same host logic over NCCL."""
import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = 10.0 + 5.0 * rank          # rank 1 is the slower one
        slowest = bench.max_over_ranks(mine, "cpu")
        rate = bench.whole_job_rate(world, 5120, 4, slowest)
        dist.barrier()
        out.put((rank, mine, slowest, rate))
    finally:
        dist.destroy_process_group()


def test_two_ranks_report_the_slowest_time_and_the_whole_job_rate():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[2] for r in res] == [15.0, 15.0]             # the slower rank's time on both
    assert res[0][3] == res[1][3] == pytest.approx(2 * 5120 * 4 / 0.015)


def test_one_rank_without_a_process_group():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(12.5, "cpu") == 12.5
    assert bench.whole_job_rate(1, 5120, 10, 20.0) == pytest.approx(5120 * 10 / 0.02)
