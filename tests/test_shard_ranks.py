"""The multi-rank exchange of one sharded stream on CPU (gloo ranks): each
rank prepares its shard's gap map from its frames and halo, the maps are
all-gathered, each rank resolves its entry gap and decides its frames. The
per-shard decisions here come from the oracle's fp32 distances (the GPU
shard kernels have their own parity tests); the concatenation over ranks must
equal the oracle's single pass."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

T, W, H, L, TAU = 157, 24, 16, 7, 0.3


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _stream():
    import oracle as O
    import synth
    fr = synth.generate(synth.medium(seed=4242).with_(width=W, height=H, frames=T, mean_scene_len=5))
    p = O.Params(W, H, tau=TAU, l_max=L)
    hist, _, keep = O.load().run(fr, p)
    return hist, keep


def _decide_from(hist, t0, n, g_entry):
    """Frames [t0, t0 + n) entered with gap g_entry (the last keep before t0
    was frame t0 - g_entry); returns (keep codes, gap after the last frame)."""
    import oracle as O
    o = O.load()
    r = t0 - g_entry
    codes = []
    for t in range(t0, t0 + n):
        if t == 0:
            code = O.KEEP_FIRST
        else:
            d = max(o.tv32(hist[t], hist[t - 1], W * H), o.tv32(hist[t], hist[max(r, 0)], W * H))
            code = O.KEEP_NOVELTY if np.float32(d) >= np.float32(TAU) else (O.KEEP_GAP if t - r >= L else O.KEEP_DROP)
        if code:
            r = t
        codes.append(code)
    return codes, t0 + n - r


def _rank(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2609_03675_gb300 import shards
    hist, _ = _stream()
    a, b, halo = shards.shard_bounds(T, world, rank, L)
    assert halo == min(a, L)
    local = hist[: b]  # this rank reads only frames [a - halo, b) below

    def prepare():
        return torch.tensor([_decide_from(local, a, b - a, g)[1] for g in range(1, L + 1)], dtype=torch.int32)

    codes = shards.sharded_decide(prepare, lambda g: _decide_from(local, a, b - a, g)[0], rank, world)
    q.put((rank, codes))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_sharded_stream_over_gloo_ranks(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = np.concatenate([out[r] for r in range(world)]).astype(np.uint8)
    _, keep = _stream()
    assert np.array_equal(got, keep)
    assert (keep == 2).any() and (keep == 1).any(), "the stream exercises both rules"


def test_entry_gaps_compose_in_order():
    from paper_2609_03675_gb300 import shards
    # three shards; identity-like maps except where noted
    maps = [[3, 3, 3], [2, 1, 3], [1, 2, 3]]
    assert shards.entry_gaps(maps) == [1, 3, 3]
    assert shards.shard_bounds(10, 3, 0, 4) == (0, 3, 0)
    assert shards.shard_bounds(10, 3, 2, 4) == (6, 10, 4)
