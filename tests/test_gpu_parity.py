"""GPU path against the oracle, element by element, on seeded synthetic streams.

Bar: integer histograms bit-exact; scores within 1e-6 relative of the
oracle's double-precision distance; keep codes identical (the decision is
taken in fp32 on both sides; frames in the tolerance band around tau_h are
reported).
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_helpers import assert_parity, oracle_run, run_stream

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_03675_gb300 import NGFF  # noqa: F401  (creating a handle fails loudly if the library is missing)


def _ngff(w, h, **kw):
    from paper_2609_03675_gb300 import NGFF
    return NGFF(w, h, **kw)


def test_tiny_stream_whole_push():
    spec = synth.tiny()
    fr = synth.generate(spec)
    p = O.Params(spec.width, spec.height)
    want = oracle_run(fr, p)
    f = _ngff(spec.width, spec.height)
    got = run_stream(f, torch.from_numpy(fr).cuda(), [spec.frames])
    band = assert_parity(got, want, p.tau, "tiny")
    # at tau_h = 0.30 the tiny stream's cuts are too small to see: first + gap keeps only
    assert list(np.flatnonzero(got[2])) == [0, 30, 60] and len(band) == 0


def test_banded_cuts_kept():
    spec = synth.tiny_banded()
    fr = synth.generate(spec)
    p = O.Params(spec.width, spec.height)
    want = oracle_run(fr, p)
    got = run_stream(_ngff(spec.width, spec.height), torch.from_numpy(fr).cuda(), [spec.frames])
    assert_parity(got, want, p.tau, "banded")
    cuts = synth.scene_starts(spec)[1:]
    assert (got[2][cuts] == 1).all()


def test_medium_stream_chunks_of_8():
    spec = synth.medium()
    fr = synth.generate(spec)
    for tau in (0.30, 0.05, 0.02):
        p = O.Params(spec.width, spec.height, tau=tau)
        want = oracle_run(fr, p)
        got = run_stream(_ngff(spec.width, spec.height, tau=tau), torch.from_numpy(fr).cuda(), [8] * 75)
        assert_parity(got, want, tau, f"medium tau={tau}")


@pytest.mark.parametrize("w,h", [(16, 1), (20, 4), (17, 13), (1, 1), (33, 7), (64, 48), (100, 3)])
@pytest.mark.parametrize("bins,l_max,tau", [(32, 30, 0.05), (1, 1, 0.3), (3, 2, 0.0), (7, 33, 0.1),
                                            (64, 5, 1.5), (256, 64, 0.02), (24, 256, 0.2)])
def test_shapes_and_params(w, h, bins, l_max, tau):
    g = np.random.default_rng(w * 1000 + h * 7 + bins + l_max)
    T = 150
    spec = synth.medium(seed=int(g.integers(1 << 30))).with_(width=w, height=h, frames=T, mean_scene_len=6)
    fr = synth.generate(spec)
    p = O.Params(w, h, bins=bins, l_max=l_max, tau=tau)
    want = oracle_run(fr, p)
    f = _ngff(w, h, bins=bins, l_max=l_max, tau=tau, max_frames_per_push=37)
    cuts = np.sort(g.choice(np.arange(1, T), size=9, replace=False))
    chunks = np.diff(np.concatenate([[0], cuts, [T]])).tolist()
    got = run_stream(f, torch.from_numpy(fr).cuda(), chunks)
    assert_parity(got, want, tau, f"{w}x{h} B={bins} L={l_max} tau={tau}")


def test_push_split_invariance_and_empty_push():
    spec = synth.medium().with_(width=96, height=64, frames=200)
    fr = synth.generate(spec)
    p = O.Params(96, 64, tau=0.05)
    want = oracle_run(fr, p)
    dev = torch.from_numpy(fr).cuda()
    f = _ngff(96, 64, tau=0.05)
    for chunks in ([200], [1] * 200, [3, 97, 1, 99], [29, 30, 31, 110]):
        f.reset()
        got = run_stream(f, dev, chunks)
        assert_parity(got, want, 0.05, f"chunks {chunks[:4]}")
    s, k = f.push(dev[:0])  # n = 0: a no-op
    assert s.numel() == 0 and k.numel() == 0


def test_reset_restarts_stream():
    spec = synth.medium().with_(width=64, height=32, frames=90)
    fr = torch.from_numpy(synth.generate(spec)).cuda()
    f = _ngff(64, 32, tau=0.05)
    a = run_stream(f, fr, [90])
    f.push(fr[:45])
    f.reset()
    assert f.frames_seen() == 0
    b = run_stream(f, fr, [90])
    for x, y in zip(a, b):
        assert np.array_equal(x, y)


def test_multistream_batch_equals_single():
    g = np.random.default_rng(5)
    S, T, w, h = 6, 120, 48, 32
    specs = [synth.medium(seed=100 + s).with_(width=w, height=h, frames=T) for s in range(S)]
    frames = [torch.from_numpy(synth.generate(sp)).cuda() for sp in specs]
    p = O.Params(w, h, tau=0.05)
    want = [oracle_run(synth.generate(sp), p) for sp in specs]
    f = _ngff(w, h, tau=0.05, max_streams=S)
    pos = [0] * S
    outs = [(torch.empty(T, dtype=torch.float32, device="cuda"), torch.empty(T, dtype=torch.uint8, device="cuda"))
            for _ in range(S)]
    while min(pos) < T:
        items = []
        for s in g.permutation(S):
            if pos[s] >= T:
                continue
            n = int(min(g.integers(0, 9), T - pos[s]))
            items.append((int(s), frames[s][pos[s]:pos[s] + n], outs[s][0][pos[s]:pos[s] + n],
                          outs[s][1][pos[s]:pos[s] + n]))
            pos[s] += n
        f.push_batch(items)
    torch.cuda.synchronize()
    f.status()
    for s in range(S):
        got_s, got_k = outs[s][0].cpu().numpy(), outs[s][1].cpu().numpy()
        ho, so, ko = want[s]
        assert np.array_equal(got_k, ko), f"stream {s}"
        assert (np.abs(got_s - so) <= 1e-6 * so).all()


def test_batch_with_host_frames_and_outputs():
    """push_batch with each descriptor's frames and outputs in device, pinned
    host or pageable host memory (the mix changes from call to call), staged
    through buffers that several calls reuse in turn, against the oracle."""
    from paper_2609_03675_gb300 import _abi
    g = np.random.default_rng(11)
    S, T, w, h = 5, 90, 48, 32
    specs = [synth.medium(seed=200 + s).with_(width=w, height=h, frames=T) for s in range(S)]
    frames_np = [synth.generate(sp) for sp in specs]
    frames_dev = [torch.from_numpy(x).cuda() for x in frames_np]
    frames_pin = [torch.from_numpy(x).pin_memory() for x in frames_np]
    p = O.Params(w, h, tau=0.05)
    want = [oracle_run(x, p) for x in frames_np]
    fb = specs[0].frame_bytes
    # staging of 40 frames: a call of up to 5 x 8 host frames fits one buffer
    f = _ngff(w, h, tau=0.05, max_streams=S, host_stage_bytes=40 * fb)
    out_dev = [(torch.zeros(T, dtype=torch.float32, device="cuda"), torch.zeros(T, dtype=torch.uint8, device="cuda"))
               for _ in range(S)]
    out_pin = [(torch.zeros(T, dtype=torch.float32).pin_memory(), torch.zeros(T, dtype=torch.uint8).pin_memory())
               for _ in range(S)]
    out_np = [(np.zeros(T, np.float32), np.zeros(T, np.uint8)) for _ in range(S)]
    # where each frame's outputs went: 0 device, 1 pinned, 2 pageable
    where = np.full((S, T), -1)
    pos = [0] * S
    while min(pos) < T:
        arr = (_abi.PushDesc * S)()
        nd = 0
        for s in g.permutation(S):
            if pos[s] >= T:
                continue
            n = int(min(g.integers(0, 9), T - pos[s]))
            a, fk, ok = pos[s], int(g.integers(0, 3)), int(g.integers(0, 3))
            d = arr[nd]
            d.stream, d.n = int(s), n
            d.frames = (frames_dev[s].data_ptr(), frames_pin[s].data_ptr(), frames_np[s].ctypes.data)[fk] + a * fb
            if ok == 0:
                d.scores_out, d.keep_out = out_dev[s][0].data_ptr() + 4 * a, out_dev[s][1].data_ptr() + a
            elif ok == 1:
                d.scores_out, d.keep_out = out_pin[s][0].data_ptr() + 4 * a, out_pin[s][1].data_ptr() + a
            else:
                d.scores_out, d.keep_out = out_np[s][0].ctypes.data + 4 * a, out_np[s][1].ctypes.data + a
            where[s, a:a + n] = ok
            pos[s] += n
            nd += 1
        f.push_batch_raw(arr, nd)
    torch.cuda.synchronize()
    f.status()
    for s in range(S):
        sc = np.select([where[s] == 0, where[s] == 1], [out_dev[s][0].cpu().numpy(), out_pin[s][0].numpy()],
                       out_np[s][0])
        kc = np.select([where[s] == 0, where[s] == 1], [out_dev[s][1].cpu().numpy(), out_pin[s][1].numpy()],
                       out_np[s][1])
        _, so, ko = want[s]
        assert np.array_equal(kc, ko), f"stream {s}: keep codes differ at {np.flatnonzero(kc != ko)[:10]}"
        assert (np.abs(sc.astype(np.float64) - so) <= 1e-6 * so).all(), f"stream {s}"
    # host frames beyond one staging buffer are refused before anything is enqueued
    big = (_abi.PushDesc * 1)()
    big[0].stream, big[0].n, big[0].frames = 0, 41, frames_pin[0].data_ptr()
    assert f._lib.cofie_ngff_push_batch(f._h, big, 1, None) == _abi.EINVAL
    assert b"staging" in f._lib.cofie_ngff_last_error(f._h)
    twice = (_abi.PushDesc * 3)()
    for i, st in enumerate((1, 3, 1)):
        twice[i].stream, twice[i].n, twice[i].frames = st, 1, frames_dev[st].data_ptr()
    assert f._lib.cofie_ngff_push_batch(f._h, twice, 3, None) == _abi.EINVAL
    assert b"appears twice" in f._lib.cofie_ngff_last_error(f._h)
    f.close()


def test_host_frames_and_host_outputs():
    spec = synth.medium().with_(width=128, height=96, frames=70)
    fr = synth.generate(spec)
    p = O.Params(128, 96, tau=0.05)
    ho, so, ko = oracle_run(fr, p)
    # staging buffers of 5 frames force several overlapped host->device pieces
    f = _ngff(128, 96, tau=0.05, host_stage_bytes=5 * spec.frame_bytes)
    pinned = torch.from_numpy(fr).pin_memory()
    scores = torch.empty(70, dtype=torch.float32).pin_memory()
    keep = torch.empty(70, dtype=torch.uint8).pin_memory()
    hist = torch.empty((70, 32), dtype=torch.int32).pin_memory()
    f.push(pinned, scores=scores, keep=keep, hist=hist)
    torch.cuda.synchronize()
    f.status()
    assert_parity((hist.numpy().view(np.uint32), scores.numpy(), keep.numpy()), (ho, so, ko), 0.05, "host")
    # pageable host memory (plain numpy) through the raw entry point
    f.reset()
    s2 = np.zeros(70, np.float32)
    k2 = np.zeros(70, np.uint8)
    f.push_raw(0, fr.ctypes.data, 70, s2.ctypes.data, k2.ctypes.data)
    torch.cuda.synchronize()
    assert np.array_equal(k2, ko)


def test_all_triples_frame_histogram():
    """A 4096x4096 frame holding every RGB triple once, through the histogram kernel (B = 256: bin = Y)."""
    v = torch.arange(1 << 24, dtype=torch.int64)
    px = torch.stack([(v >> 16) & 255, (v >> 8) & 255, v & 255], -1).to(torch.uint8).reshape(1, 4096, 4096, 3)
    o = O.load()
    for bins in (256, 32):
        want = o.histogram(px.numpy()[0], O.Params(4096, 4096, bins=bins))
        f = _ngff(4096, 4096, bins=bins)
        _, _, h = f.push(px.cuda(), return_hist=True)
        torch.cuda.synchronize()
        assert np.array_equal(h.cpu().numpy()[0].view(np.uint32), want)


def test_histogram_rows_cleared_between_pushes():
    """Pushes that return their histograms and pushes that do not, small
    (fused selection kernel) and large (separate kernels), interleaved on one
    stream and across two handles' streams, all match the oracle."""
    spec = synth.medium(seed=41).with_(width=80, height=48, frames=400, mean_scene_len=12)
    fr = synth.generate(spec)
    ho, so, ko = oracle_run(fr, O.Params(80, 48, tau=0.05))
    dev = torch.from_numpy(fr).cuda()
    f = _ngff(80, 48, tau=0.05, max_streams=2)
    chunks = [5, 130, 64, 65, 1, 100, 8, 27]  # sums to 400
    want_hist = [True, False, False, True, False, True, True, False]
    got_s, got_k = [], []
    off = 0
    for c, wh in zip(chunks, want_hist):
        if wh:
            s, k, h = f.push(dev[off:off + c], return_hist=True)
            torch.cuda.synchronize()
            assert np.array_equal(h.cpu().numpy().view(np.uint32), ho[off:off + c])
        else:
            s, k = f.push(dev[off:off + c])
        # a second stream interleaved, always without histograms
        f.push(dev[off:off + c], stream=1)
        got_s.append(s)
        got_k.append(k)
        off += c
    torch.cuda.synchronize()
    f.status()
    assert np.array_equal(torch.cat(got_k).cpu().numpy(), ko)
    s = torch.cat(got_s).cpu().numpy().astype(np.float64)
    assert np.all(np.abs(s - so) <= 1e-6 * so)
