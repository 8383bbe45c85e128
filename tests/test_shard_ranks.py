"""The multi-rank exchange of one sharded stream (gloo ranks): each rank holds
only its shard and a halo of min(a, L_max) frames before it, prepares its
shard's gap map, the maps are all-gathered, each rank resolves its entry gap
and decides its frames. On CPU the per-shard decisions come from the oracle's
fp32 distances on the rank's own frames (a stand-in for the library); where a
GPU is present each rank runs the library's own cofie_ngff_shard_prepare and
_commit through shards.sharded_push, every rank on its own handle. The
concatenation over ranks must equal the oracle's single pass."""
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


def _spec():
    import synth
    return synth.medium(seed=4242).with_(width=W, height=H, frames=T, mean_scene_len=5)


def _single_pass():
    import oracle as O
    import synth
    _, _, keep = O.load().run(synth.generate(_spec()), O.Params(W, H, tau=TAU, l_max=L))
    return keep


def _decide_from(hist, lo, t0, n, g_entry):
    """Frames [t0, t0 + n) entered with gap g_entry (the last keep before t0
    was frame t0 - g_entry), from the histograms of frames [lo, t0 + n) only
    (hist[i] is frame lo + i); returns (keep codes, gap after the last frame)."""
    import oracle as O
    o = O.load()
    r = t0 - g_entry
    codes = []
    for t in range(t0, t0 + n):
        if t == 0:
            code = O.KEEP_FIRST
        else:
            d = max(o.tv32(hist[t - lo], hist[t - 1 - lo], W * H), o.tv32(hist[t - lo], hist[max(r, 0) - lo], W * H))
            code = O.KEEP_NOVELTY if np.float32(d) >= np.float32(TAU) else (O.KEEP_GAP if t - r >= L else O.KEEP_DROP)
        if code:
            r = t
        codes.append(code)
    return codes, t0 + n - r


def _rank(rank, world, port, q, on_gpu):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle as O
    import synth
    from paper_2609_03675_gb300 import shards
    a, b, halo = shards.shard_bounds(T, world, rank, L)
    assert halo == min(a, L)
    lo, hi = shards.shard_frames(T, world, rank, L)
    local = synth.generate(_spec(), lo, hi)  # this rank's frames only: the halo, then the shard
    if on_gpu:
        from paper_2609_03675_gb300 import NGFF
        torch.cuda.set_device(0)
        f = NGFF(W, H, tau=TAU, l_max=L)
        _, keep = shards.sharded_push(f, torch.from_numpy(local).cuda(), T, rank, world)
        torch.cuda.synchronize()
        f.status()
        codes = keep.cpu().tolist()
        f.close()
    else:
        hist = O.load().run(local, O.Params(W, H, tau=TAU, l_max=L))[0]

        def prepare():
            return torch.tensor([_decide_from(hist, lo, a, b - a, g)[1] for g in range(1, L + 1)], dtype=torch.int32)

        codes = shards.sharded_decide(prepare, lambda g: _decide_from(hist, lo, a, b - a, g)[0], rank, world)
    q.put((rank, codes))
    dist.barrier()
    dist.destroy_process_group()


def _run_ranks(world, on_gpu):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q, on_gpu)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=300) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = np.concatenate([out[r] for r in range(world)]).astype(np.uint8)
    keep = _single_pass()
    assert np.array_equal(got, keep)
    assert (keep == 2).any() and (keep == 1).any(), "the stream exercises both rules"
    if on_gpu:  # the sharded stream closed from its shards' keep codes
        import oracle as O
        from paper_2609_03675_gb300 import NGFF
        f = NGFF(W, H, tau=TAU, l_max=L)
        idx = f.candidates_from_keep(torch.from_numpy(got).cuda()).cpu().numpy().astype(np.uint32)
        assert np.array_equal(idx, O.load().candidates(keep, 4))
        f.close()


@pytest.mark.parametrize("world", [2, 3])
def test_sharded_stream_over_gloo_ranks(world):
    _run_ranks(world, on_gpu=False)


@pytest.mark.gpu
@pytest.mark.parametrize("world", [2, 3])
def test_sharded_stream_over_gloo_ranks_on_the_library(world):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    _run_ranks(world, on_gpu=True)


def test_shard_frames_are_the_halo_and_the_shard():
    from paper_2609_03675_gb300 import shards
    for world in (1, 2, 3, 5):
        covered = []
        for r in range(world):
            a, b, halo = shards.shard_bounds(T, world, r, L)
            lo, hi = shards.shard_frames(T, world, r, L)
            assert (lo, hi) == (a - halo, b) and hi - lo <= b - a + L
            covered += list(range(a, b))
        assert covered == list(range(T))


def test_entry_gaps_compose_in_order():
    from paper_2609_03675_gb300 import shards
    # three shards; identity-like maps except where noted
    maps = [[3, 3, 3], [2, 1, 3], [1, 2, 3]]
    assert shards.entry_gaps(maps) == [1, 3, 3]
    assert shards.shard_bounds(10, 3, 0, 4) == (0, 3, 0)
    assert shards.shard_bounds(10, 3, 2, 4) == (6, 10, 4)
