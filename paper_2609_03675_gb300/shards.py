"""One stream split across ranks: the host side of the single exchange step.

The rule of Sec. 3.2 depends on the past only through the gap t - r(t) in
[1, L_max] and the histograms of the L_max frames before t. So a contiguous
shard [a, b) of a stream can be prepared on its own rank from its frames plus
a halo of min(a, L_max) frames before it (cofie_ngff_shard_prepare), giving
its gap map: for every entry gap g, the gap after its last frame. The maps are
the only data the ranks exchange (L_max small integers each, one all-gather);
every rank then composes the maps of the shards before it, in stream order,
to find its own entry gap, and decides its frames (cofie_ngff_shard_commit).
Shard 0 holds the stream's first frame, which is kept whatever the entry.
"""
from __future__ import annotations

from typing import Callable, Sequence

import torch
import torch.distributed as dist


def shard_bounds(T: int, world: int, rank: int, l_max: int) -> tuple[int, int, int]:
    """(a, b, halo) of rank's contiguous shard of a T-frame stream: frames
    [a, b), prepared from frames [a - halo, b)."""
    a, b = T * rank // world, T * (rank + 1) // world
    return a, b, min(a, l_max)


def entry_gaps(maps: Sequence[Sequence[int]]) -> list[int]:
    """Entry gap of every shard, from the gap maps of all shards in stream
    order (maps[i][g - 1]: the gap after shard i's last frame when it is
    entered with gap g)."""
    gaps = [1]
    for m in maps[:-1]:
        gaps.append(int(m[gaps[-1] - 1]))
    return gaps


def exchange_maps(local_map: torch.Tensor, world: int, group=None) -> list[torch.Tensor]:
    """All-gathers every rank's gap map (an int tensor of L_max entries)."""
    t = local_map.to(torch.int32).reshape(-1)
    if dist.get_backend(group) == "nccl":
        t = t.cuda()
    out = [torch.empty_like(t) for _ in range(world)]
    dist.all_gather(out, t, group=group)
    return [o.cpu() for o in out]


def sharded_decide(prepare: Callable[[], torch.Tensor], commit: Callable[[int], object], rank: int, world: int,
                   group=None):
    """prepare() -> this rank's gap map; commit(entry_gap) -> its decisions.
    One all-gather of the maps between the two."""
    maps = exchange_maps(prepare(), world, group)
    return commit(entry_gaps([m.tolist() for m in maps])[rank])


def shard_frames(T: int, world: int, rank: int, l_max: int) -> tuple[int, int]:
    """The frames [lo, hi) a rank must hold for its shard of a T-frame stream:
    its halo of min(a, L_max) frames, then its own frames [a, b)."""
    a, b, halo = shard_bounds(T, world, rank, l_max)
    return a - halo, b


def sharded_push(f, local_frames: torch.Tensor, T: int, rank: int, world: int, group=None, stream: int = 0):
    """Decides rank's shard of a T-frame stream. local_frames holds only the
    frames shard_frames() names (the halo, then the shard: b - a + halo
    frames on this rank's device), so per-rank memory is the shard plus
    L_max frames. Returns (scores, keep) of frames [a, b)."""
    a, b, halo = shard_bounds(T, world, rank, f.l_max)
    if local_frames.shape[0] != b - a + halo:
        raise ValueError(f"rank {rank} needs frames [{a - halo}, {b}) ({b - a + halo} frames), "
                         f"got {local_frames.shape[0]}")
    return sharded_decide(lambda: f.shard_prepare(local_frames, n_halo=halo, t0=a, stream=stream),
                          lambda g: f.shard_commit(g, b - a, stream=stream), rank, world, group)
