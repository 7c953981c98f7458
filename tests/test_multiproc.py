"""The bench's multi-rank bookkeeping on CPU ranks (gloo, world size 2): every rank runs
a replica, the job's step time is the maximum over ranks and the value counts all ranks'
tokens."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        # rank r reports step times (10 + r, 3 - r) ms; the job sees the slowest of each
        total, kernel = bench.max_over_ranks([10.0 + rank, 3.0 - rank], world)
        value = bench.job_value(world, 65536, total)
        dist.barrier()
        q.put((rank, total, kernel, value))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_value_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, total, kernel, value in out:
        assert total == 11.0 and kernel == 3.0
        assert value == pytest.approx(2 * 65536 / 11e-3)


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks([1.5, 2.5], 1) == [1.5, 2.5]
    assert bench.job_value(1, 1000, 2.0) == pytest.approx(5e5)
