"""Checkpoint/resume of a stream and sharding one stream across handles.

Both rest on the same fact (Sec. 3.2, Eqs. 3-5): a frame's decision depends
on the past only through the gap t - r(t) in [1, L_max] and the histograms
of the L_max frames before it. Saved and restored streams, and shards
prepared independently (here on separate handles, in reverse order) and
chained through their gap maps, must give the oracle's single-pass result."""
import numpy as np
import pytest
import torch

import oracle as O
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _stream(T=300, w=64, h=48, seed=51, mean=9):
    spec = synth.medium(seed=seed).with_(width=w, height=h, frames=T, mean_scene_len=mean)
    return spec, synth.generate(spec)


@pytest.mark.parametrize("buf_on_device", [False, True])
def test_save_restore_continues_the_stream(buf_on_device):
    from paper_2609_03675_gb300 import NGFF
    spec, fr = _stream()
    _, so, ko = O.load().run(fr, O.Params(spec.width, spec.height, tau=0.05))
    dev = torch.from_numpy(fr).cuda()
    a = NGFF(spec.width, spec.height, tau=0.05)
    s1, k1 = a.push(dev[:117])
    out = torch.empty(0)
    if buf_on_device:
        out = torch.empty(a._lib.cofie_ngff_state_bytes(a._h), dtype=torch.uint8, device="cuda")
        state = a.state_save(out=out)
    else:
        state = a.state_save()
    a.close()
    b = NGFF(spec.width, spec.height, tau=0.05, max_streams=3)
    b.state_load(state, stream=2)
    assert b.frames_seen(2) == 117
    s2, k2 = b.push(dev[117:], stream=2)
    torch.cuda.synchronize()
    b.status()
    assert np.array_equal(torch.cat([k1, k2]).cpu().numpy(), ko)
    assert np.all(np.abs(torch.cat([s1, s2]).cpu().numpy().astype(np.float64) - so) <= 1e-6 * so)


def test_restore_refuses_another_shape():
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    spec, fr = _stream(T=10)
    a = NGFF(spec.width, spec.height)
    a.push(torch.from_numpy(fr).cuda())
    state = a.state_save()
    for kw in ({"bins": 16}, {"l_max": 29}):
        with pytest.raises(NGFFError) as e:
            NGFF(spec.width, spec.height, **kw).state_load(state)
        assert e.value.code == _abi.EINVAL
    bad = state.clone()
    bad[0] ^= 0xFF
    with pytest.raises(NGFFError):
        NGFF(spec.width, spec.height).state_load(bad)


@pytest.mark.parametrize("cuts,l_max", [([80, 81, 190], 30), ([10, 40, 41, 230], 30), ([5, 60, 61, 150], 7),
                                        ([100, 200], 256)])
def test_shards_prepared_independently_and_chained(cuts, l_max):
    from paper_2609_03675_gb300 import NGFF
    T = 300
    spec, fr = _stream(T=T, seed=52)
    tau = 0.05
    _, so, ko = O.load().run(fr, O.Params(spec.width, spec.height, tau=tau, l_max=l_max))
    dev = torch.from_numpy(fr).cuda()
    bounds = [0] + cuts + [T]
    shards = list(zip(bounds[:-1], bounds[1:]))
    handles, maps = {}, {}
    for a, b in reversed(shards):  # any order: each shard needs only its frames and halo
        f = NGFF(spec.width, spec.height, tau=tau, l_max=l_max)
        halo = min(a, l_max)
        maps[a] = f.shard_prepare(dev[a - halo:b], n_halo=halo, t0=a).numpy()
        handles[a] = f
    gap, outs = 1, []
    for a, b in shards:
        s, k = handles[a].shard_commit(gap, b - a)
        outs.append((s, k))
        gap = int(maps[a][gap - 1])
    torch.cuda.synchronize()
    for f in handles.values():
        f.status()
    keep = torch.cat([k for _, k in outs]).cpu().numpy()
    score = torch.cat([s for s, _ in outs]).cpu().numpy().astype(np.float64)
    assert np.array_equal(keep, ko)
    assert np.all(np.abs(score - so) <= 1e-6 * so)
    # the last shard's handle is left exactly as a single pass would leave it
    # (header, gap and ring); each shard's retention record holds its own
    # retained frames, and together they are the single pass's record
    single = NGFF(spec.width, spec.height, tau=tau, l_max=l_max)
    single.push(dev)
    torch.cuda.synchronize()
    one = single.state_save().numpy()
    ring_end = 64 + l_max * 32 * 4
    assert np.array_equal(handles[shards[-1][0]].state_save().numpy()[:ring_end], one[:ring_end])
    record = (lambda st: np.unpackbits(st[ring_end:], bitorder="little"))
    union = np.zeros_like(record(one))
    for a, b in shards:
        r = record(handles[a].state_save().numpy())
        assert np.array_equal(np.flatnonzero(r), a + np.flatnonzero(ko[a:b])), f"shard [{a}, {b})"
        union |= r
    assert np.array_equal(union, record(one))
    assert np.array_equal(np.flatnonzero(record(one)), np.flatnonzero(ko))
    # the sharded stream closed from its shards' keep codes
    idx = handles[shards[-1][0]].candidates_from_keep(torch.cat([k for _, k in outs]))
    assert np.array_equal(idx.cpu().numpy().astype(np.uint32), O.load().candidates(ko, 4))
