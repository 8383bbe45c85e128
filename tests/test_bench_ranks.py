"""The multi-rank host logic of bench.py on CPU: world_size-2 gloo ranks.

Each rank filters its own stream (distinct seeds), the timing is the max over
ranks, and the whole-job rate counts every rank's frames over that time."""
import os
import socket

import pytest
import torch.multiprocessing as mp

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


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


def _bench(args, env=None):
    import json
    import subprocess
    import sys
    e = dict(os.environ)
    e.update(env or {})
    r = subprocess.run([sys.executable, os.path.join(REPO, "bench.py"), *args], capture_output=True, text=True,
                       timeout=600, env=e, cwd=REPO)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    return [json.loads(ln) for ln in lines]


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` (the oracle on host cores) prints one JSON
    line with the benchmark's keys, a cpu_baseline describing the run, and an
    e2e object with no host-device bytes."""
    (d,) = _bench(["--impl", "reference", "--steps", "1", "--warmup", "0"])
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "frames/s"
    for key in ("metric", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling", "dtype", "data"):
        assert key in d, key
    assert d["vs_baseline"] is None and d["higher_is_better"] is True and d["steps"] == 1
    assert "workload" in d["config"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_do_no_work():
    """Under torchrun only rank 0 runs the reference arm; the others exit 0 silently."""
    assert _bench(["--impl", "reference", "--steps", "1", "--warmup", "0"], {"RANK": "1", "WORLD_SIZE": "2"}) == []
