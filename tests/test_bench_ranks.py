"""The multi-rank host logic of bench.py on CPU: world_size-2 gloo ranks.

Each rank filters its own stream (distinct seeds), the timing is the max over
ranks, and the whole-job rate counts every rank's frames over that time."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    r, w, local = bench.dist_env()
    ms = bench.max_over_ranks(10.0 + 5.0 * rank, device="cpu")  # rank 1 is the slow one
    rate = bench.whole_job_rate(3600, w, ms / 1e3)
    q.put((r, w, local, bench.stream_seed(r), ms, rate))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_max_time_and_whole_job_rate():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    (r0, w0, l0, s0, ms0, v0), (r1, w1, l1, s1, ms1, v1) = out
    assert (r0, r1, w0, w1, l0, l1) == (0, 1, 2, 2, 0, 1)
    assert s0 != s1, "ranks must filter independently seeded streams"
    assert ms0 == ms1 == 15.0, "timing is the max over ranks"
    assert v0 == v1 == pytest.approx(2 * 3600 / 0.015)


def test_single_process_needs_no_group():
    import bench
    assert bench.max_over_ranks(3.5, device="cpu") == 3.5
    assert bench.whole_job_rate(100, 1, 0.5) == 200.0
