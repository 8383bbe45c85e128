"""Closing a stream through its retention record: cofie_ngff_candidates(h,
stream, idx_out, cap, &m) after pushes, against the oracle's candidate set
(last frame, M_min uniform fill; the retention safeguards of Sec. 3.2) of the
oracle's keep codes for the same prefix.

The keep codes of a prefix are those of the whole stream cut at the prefix
(decisions are causal), so one oracle run per stream serves every prefix.
The full-size streams (1080p in pieces, the 32 serving streams) are closed in
tests/test_gpu_fullsize.py."""
import ctypes

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


def _close_abi(f, stream, cap, device_m: bool):
    """The C entry point called directly: device indices, m in device or host memory."""
    idx = torch.full((max(cap, 1),), -7, dtype=torch.int32, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    if device_m:
        m_dev = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        rc = f._lib.cofie_ngff_candidates(f._h, stream, idx.data_ptr(), cap, m_dev.data_ptr(), st)
        assert rc == 0, f._lib.cofie_ngff_last_error(f._h)
        m = int(m_dev.item())
    else:
        mh = ctypes.c_uint32(0xFFFFFFFF)
        rc = f._lib.cofie_ngff_candidates(f._h, stream, idx.data_ptr(), cap, ctypes.addressof(mh), st)
        assert rc == 0, f._lib.cofie_ngff_last_error(f._h)
        m = mh.value
    return m, idx.cpu().numpy().view(np.uint32)


@pytest.mark.parametrize("tau", [0.30, 0.05])
def test_medium_stream_in_chunks_of_8_closed_at_prefixes(tau):
    """The medium stream (600 frames of 448x448) pushed 8 frames at a time,
    closed after several of the pushes, with the count read from device and
    from host memory."""
    from paper_2609_03675_gb300 import NGFF
    spec = synth.medium()
    fr = synth.generate(spec)
    dev = torch.from_numpy(fr).cuda()
    o = O.load()
    _, _, ko = o.run(fr, O.Params(spec.width, spec.height, tau=tau))
    f = NGFF(spec.width, spec.height, tau=tau)
    close_at = {8, 16, 24, 64, 304, 600}
    for t in range(0, spec.frames, 8):
        f.push(dev[t:t + 8])
        T = t + 8
        if T in close_at:
            want = o.candidates(ko[:T], 4)
            for device_m in (True, False):
                m, idx = _close_abi(f, 0, T, device_m)
                assert m == want.size and np.array_equal(idx[:m], want), f"T={T} tau={tau} device_m={device_m}"
    f.status()
    assert f.frames_seen() == spec.frames
    f.close()


def test_short_prefixes_and_the_uniform_fill():
    """Prefixes of 1..12 frames pushed one at a time, at a threshold no frame
    reaches (only the first frame is retained before the gap rule), for
    M_min 1..6: the fill decides most of S_c."""
    from paper_2609_03675_gb300 import NGFF
    spec = synth.medium(seed=41).with_(width=64, height=48, frames=12)
    fr = synth.generate(spec)
    dev = torch.from_numpy(fr).cuda()
    o = O.load()
    for m_min in range(1, 7):
        for l_max in (30, 5, 0):
            _, _, ko = o.run(fr, O.Params(spec.width, spec.height, tau=2.0, l_max=l_max))
            f = NGFF(spec.width, spec.height, tau=2.0, l_max=l_max, m_min=m_min)
            for T in range(1, spec.frames + 1):
                f.push(dev[T - 1:T])
                got = f.candidates(0).cpu().numpy().astype(np.uint32)
                assert np.array_equal(got, o.candidates(ko[:T], m_min)), f"T={T} M_min={m_min} L_max={l_max}"
            f.close()


def test_cap_smaller_than_the_set_reports_the_full_count():
    from paper_2609_03675_gb300 import NGFF
    spec = synth.medium(seed=42).with_(width=64, height=48, frames=300, mean_scene_len=4)
    fr = synth.generate(spec)
    f = NGFF(spec.width, spec.height, tau=0.02)
    f.push(torch.from_numpy(fr).cuda())
    _, _, ko = O.load().run(fr, O.Params(spec.width, spec.height, tau=0.02))
    want = O.load().candidates(ko, 4)
    assert want.size > 40
    m, idx = _close_abi(f, 0, 40, True)
    assert m == want.size and np.array_equal(idx[:40], want[:40])
    assert (idx[40:] == np.uint32(0xFFFFFFF9)).all(), "nothing is written past cap"
    m0, _ = _close_abi(f, 0, 0, True)  # cap 0: the count alone
    assert m0 == want.size
    f.close()


def test_streams_of_a_batch_reset_and_resumed_state():
    """Several streams of one handle pushed through the batched call, one of
    them reset and restarted (its record empties), one saved and resumed on
    another handle (the record travels with the state)."""
    from paper_2609_03675_gb300 import NGFF
    o = O.load()
    specs = [synth.medium(seed=50 + s).with_(width=96, height=64, frames=160, mean_scene_len=6) for s in range(3)]
    frs = [synth.generate(sp) for sp in specs]
    devs = [torch.from_numpy(x).cuda() for x in frs]
    kos = [o.run(x, O.Params(96, 64, tau=0.05))[2] for x in frs]
    f = NGFF(96, 64, tau=0.05, max_streams=3)
    sizes = [5, 1, 8, 3, 7, 2, 8, 6]
    pos = [0, 0, 0]
    i = 0
    while min(pos) < 160:
        items = []
        for s in range(3):
            n = min(sizes[(i + s) % len(sizes)], 160 - pos[s])
            if n:
                items.append((s, devs[s][pos[s]:pos[s] + n], None, None))
                pos[s] += n
        f.push_batch(items)
        i += 1
        if i % 7 == 0:
            for s in range(3):
                got = f.candidates(s).cpu().numpy().astype(np.uint32)
                assert np.array_equal(got, o.candidates(kos[s][:pos[s]], 4)), f"stream {s} at {pos[s]}"
    # reset stream 1 and push its first 20 frames again: only those count
    f.reset(1)
    assert f.candidates(1).numel() == 0
    f.push(devs[1][:20], 1)
    assert np.array_equal(f.candidates(1).cpu().numpy().astype(np.uint32), o.candidates(kos[1][:20], 4))
    # stream 2 saved at 160 frames, resumed on another handle with 100 more frames of its stream
    spec_long = specs[2].with_(frames=260)
    fr_long = synth.generate(spec_long)
    ko_long = o.run(fr_long, O.Params(96, 64, tau=0.05))[2]
    state = f.state_save(2)
    g = NGFF(96, 64, tau=0.05)
    g.state_load(state)
    g.push(torch.from_numpy(fr_long[160:]).cuda())
    assert np.array_equal(g.candidates(0).cpu().numpy().astype(np.uint32), o.candidates(ko_long, 4))
    f.status()
    g.status()
    f.close()
    g.close()


def test_signals_and_scene_changes_record_their_keeps():
    """The low-res and dHash signals (their own first stage), scene changes,
    and L_max = 0: the record holds what each rule retained."""
    from oracle import scd_oracle as SC
    from oracle import signals_oracle as SO
    from paper_2609_03675_gb300 import NGFF, _abi
    spec = synth.medium(seed=61).with_(width=128, height=96, frames=400, mean_scene_len=8)
    fr = synth.generate(spec)
    dev = torch.from_numpy(fr).cuda()
    o = O.load()
    cases = []
    for sig, tau in ((_abi.SIGNAL_LOWRES, 0.02), (_abi.SIGNAL_DHASH, 0.05)):
        ko = SO.run(fr, O.Params(spec.width, spec.height, tau=tau), sig)[2]
        cases.append((dict(signal=sig, tau=tau), ko))
    hist = o.run(fr, O.Params(spec.width, spec.height))[0]
    cases.append((dict(signal=_abi.SIGNAL_SCD, tau=0.30, scd_cut=0.08, scd_gradual=0.02),
                  SC.select(hist, O.Params(spec.width, spec.height, tau=0.30), 0.08, 0.02)[1]))
    cases.append((dict(l_max=0, tau=0.04), o.select(hist, O.Params(spec.width, spec.height, tau=0.04, l_max=0))[1]))
    for kw, ko in cases:
        f = NGFF(spec.width, spec.height, **kw)
        _, k = f.push(dev[:150])
        got = f.candidates(0).cpu().numpy().astype(np.uint32)
        assert np.array_equal(got, o.candidates(ko[:150], 4)), kw
        _, k2 = f.push(dev[150:])
        assert np.array_equal(torch.cat([k, k2]).cpu().numpy(), ko), kw
        got = f.candidates(0).cpu().numpy().astype(np.uint32)
        assert np.array_equal(got, o.candidates(ko, 4)), kw
        f.close()


def test_captured_push_and_close_replayed():
    """A push of 8 frames and the close that follows it, captured into one
    CUDA graph: every launch closes the longer prefix (T is read on the
    device)."""
    from paper_2609_03675_gb300 import NGFF
    spec = synth.medium(seed=71).with_(width=96, height=64, frames=96, mean_scene_len=5)
    fr = synth.generate(spec)
    dev = torch.from_numpy(fr).cuda()
    ko = O.load().run(fr, O.Params(96, 64, tau=0.05))[2]
    f = NGFF(96, 64, tau=0.05)
    buf = torch.empty_like(dev[:8])
    idx = torch.empty(spec.frames, dtype=torch.int32, device="cuda")
    m = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        f.push(buf)
        f.candidates_raw(0, idx.data_ptr(), spec.frames, m.data_ptr())
    f.reset()
    for t in range(0, spec.frames, 8):
        buf.copy_(dev[t:t + 8])
        g.replay()
        want = O.load().candidates(ko[:t + 8], 4)
        got = idx[: int(m.item())].cpu().numpy().astype(np.uint32)
        assert np.array_equal(got, want), f"T={t + 8}"
    f.status()
    f.close()


def test_stream_past_its_record():
    """max_stream_frames = 64: a close after 70 frames is refused on the host
    (COFIE_EINVAL); a captured close replayed after them writes m = 0 and
    cofie_ngff_status reports COFIE_EDEVICE; after a reset the stream closes
    normally again."""
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    spec = synth.medium(seed=72).with_(width=64, height=48, frames=70)
    fr = synth.generate(spec)
    dev = torch.from_numpy(fr).cuda()
    f = NGFF(64, 48, tau=0.05, max_stream_frames=64)
    idx = torch.empty(80, dtype=torch.int32, device="cuda")
    m = torch.full((1,), 99, dtype=torch.int32, device="cuda")
    g = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        f.candidates_raw(0, idx.data_ptr(), 80, m.data_ptr())
    f.push(dev[:64])
    ko = O.load().run(fr, O.Params(64, 48, tau=0.05))[2]
    assert np.array_equal(f.candidates(0).cpu().numpy().astype(np.uint32), O.load().candidates(ko[:64], 4))
    f.push(dev[64:])
    with pytest.raises(NGFFError) as e:
        f.candidates(0)
    assert e.value.code == _abi.EINVAL
    g.replay()
    with pytest.raises(NGFFError) as e:
        f.status()
    assert e.value.code == _abi.EDEVICE
    assert int(m.item()) == 0
    f.reset()
    f.push(dev[:10])
    assert np.array_equal(f.candidates(0).cpu().numpy().astype(np.uint32), O.load().candidates(ko[:10], 4))
    f.status()
    f.close()


@pytest.mark.parametrize("m_min", [4, 5000])
def test_long_stream_crosses_record_tiles(m_min):
    """40,000 frames (the record is compacted 32,768 frames per pass of the
    closing kernel) closed at prefixes on both sides of a pass boundary, with
    a small M_min and with one larger than the retained set (the uniform fill
    over many record words)."""
    from paper_2609_03675_gb300 import NGFF
    T = 40_000
    spec = synth.medium(seed=81).with_(width=16, height=16, frames=T, mean_scene_len=30)
    fr = synth.generate(spec)
    o = O.load()
    _, _, ko = o.run(fr, O.Params(16, 16, tau=0.35, l_max=45))
    f = NGFF(16, 16, tau=0.35, l_max=45, m_min=m_min, max_frames_per_push=4096)
    dev = torch.from_numpy(fr).cuda()
    pos = 0
    for close in (32_767, 32_768, 32_769, 40_000):
        while pos < close:
            n = min(4096, close - pos)
            f.push(dev[pos:pos + n])
            pos += n
        got = f.candidates(0).cpu().numpy().astype(np.uint32)
        want = o.candidates(ko[:close], m_min)
        assert np.array_equal(got, want), f"T={close} M_min={m_min}"
    f.status()
    assert (ko != 0).sum() < 5000, "the fill case must exercise the uniform frames"
    f.close()


def test_full_batch_of_64_streams():
    """The most streams one batched call takes (64), each pushing 0-9 frames
    per call in a shuffled descriptor order, with the scene-change signal so
    that every rule of the walk runs; every stream's keep codes, scores and
    candidate set against the oracle's."""
    from oracle import scd_oracle as SC
    from paper_2609_03675_gb300 import NGFF, _abi
    g = np.random.default_rng(64)
    S, T, w, h = _abi.MAX_BATCH, 60, 32, 16
    o = O.load()
    frs = [synth.generate(synth.medium(seed=900 + s).with_(width=w, height=h, frames=T, mean_scene_len=4))
           for s in range(S)]
    want = []
    for fr in frs:
        hist = o.run(fr, O.Params(w, h))[0]
        want.append(SC.select(hist, O.Params(w, h, tau=0.2, l_max=9), 0.15, 0.05))
    f = NGFF(w, h, tau=0.2, l_max=9, signal=_abi.SIGNAL_SCD, scd_cut=0.15, scd_gradual=0.05, max_streams=S)
    devs = [torch.from_numpy(x).cuda() for x in frs]
    sc = torch.zeros((S, T), dtype=torch.float32, device="cuda")
    kp = torch.full((S, T), 255, dtype=torch.uint8, device="cuda")
    pos = [0] * S
    while min(pos) < T:
        items = []
        for s in g.permutation(S):
            s = int(s)
            n = int(min(g.integers(0, 10), T - pos[s]))
            items.append((s, devs[s][pos[s]:pos[s] + n], sc[s, pos[s]:pos[s] + n], kp[s, pos[s]:pos[s] + n]))
            pos[s] += n
        f.push_batch(items)
    torch.cuda.synchronize()
    f.status()
    ks, ss = kp.cpu().numpy(), sc.cpu().numpy().astype(np.float64)
    for s in range(S):
        so, ko = want[s]
        assert np.array_equal(ks[s], ko), f"stream {s}"
        assert (np.abs(ss[s] - so) <= 1e-6 * so).all(), f"stream {s}"
        got = f.candidates(s).cpu().numpy().astype(np.uint32)
        assert np.array_equal(got, o.candidates(ko, 4)), f"stream {s}"
    assert any((w_[1] == SC.KEEP_SCENE).any() for w_ in want), "scene changes occur"
    f.close()
