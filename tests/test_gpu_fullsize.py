"""Full-size parity: the 1080p, 720p rare-event and 32-stream serving workloads.

Every frame's histogram, score and keep code is compared with the oracle
(its histogram routine mapped over host threads, then its selection rule),
on the same seeded bytes, in the launch configuration the benchmark times.
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_helpers import assert_parity, run_stream

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _pinned_stream(spec):
    buf = torch.empty((spec.frames, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=buf.data_ptr())
    return buf


def _oracle(buf, spec, taus):
    o = O.load()
    p = O.Params(spec.width, spec.height)
    hist = o.histograms_parallel(buf.data_ptr(), spec.frames, p)
    return hist, {tau: o.select(hist, O.Params(spec.width, spec.height, tau=tau)) for tau in taus}


def test_hd1080_whole_stream_push():
    from paper_2609_03675_gb300 import NGFF
    spec = synth.hd1080()
    buf = _pinned_stream(spec)
    dev = buf.cuda()
    taus = (0.30, 0.05)
    hist_o, sel = _oracle(buf, spec, taus)
    for tau in taus:
        f = NGFF(spec.width, spec.height, tau=tau, max_frames_per_push=spec.frames)
        got = run_stream(f, dev, [spec.frames])
        band = assert_parity(got, (hist_o, *sel[tau]), tau, f"1080p tau={tau}")
        print(f"1080p tau={tau}: kept {int((got[2] != 0).sum())}/{spec.frames}, band frames {list(band)}")
        # close the prefix and gather the encoder's input
        idx = f.candidates(0)  # the stream's own retention record
        want_idx = O.load().candidates(sel[tau][1], 4)
        assert np.array_equal(idx.cpu().numpy().astype(np.uint32), want_idx)
        out = f.gather(dev, idx)
        torch.cuda.synchronize()
        f.status()
        assert torch.equal(out.cpu(), buf[torch.from_numpy(want_idx.astype(np.int64))])
        del out
        f.close()
    # the same stream pushed in pieces and closed after each (Sec. 3.2 closing
    # safeguards on the stream's own retention record)
    f = NGFF(spec.width, spec.height, tau=0.30, max_frames_per_push=1600)
    off = 0
    for n in (1, 2, 997, 1000, 1600):
        f.push(dev[off:off + n])
        off += n
        idx = f.candidates(0).cpu().numpy().astype(np.uint32)
        assert np.array_equal(idx, O.load().candidates(sel[0.30][1][:off], 4)), f"1080p prefix {off}"
    f.status()
    f.close()
    del buf
    # every scene cut of the textured stream moves the histogram past tau = 0.30
    cuts = synth.scene_starts(spec)[1:]
    got30 = sel[0.30][1]
    print(f"1080p: {len(cuts)} cuts, {int((got30[cuts] != 0).sum())} retained at tau 0.30")


def test_hd1080_without_gap_and_with_scene_changes():
    """The two other rules the benchmark times on the 1080p stream
    (`--l-max 0`, `--signal 3`): no forced retention, walked in frame order
    (the windowed walk), and scene-change detection + H-diff (twin comparison
    over several 4096-frame scan tiles), against the oracle's rules on the
    oracle's histograms; keep codes exact, scores within the fp32 bound. The
    scene-change thresholds sit inside the stream's adjacent-difference
    distribution so that cuts and gradual runs both occur."""
    from oracle import scd_oracle as SC
    from paper_2609_03675_gb300 import NGFF, _abi
    spec = synth.hd1080()
    buf = _pinned_stream(spec)
    dev = buf.cuda()
    o = O.load()
    hist_o = o.histograms_parallel(buf.data_ptr(), spec.frames, O.Params(spec.width, spec.height))
    del buf
    # L_max = 0
    p0 = O.Params(spec.width, spec.height, tau=0.30, l_max=0)
    so, ko = o.select(hist_o, p0)
    f = NGFF(spec.width, spec.height, tau=0.30, l_max=0, max_frames_per_push=spec.frames)
    assert_parity(run_stream(f, dev, [spec.frames]), (hist_o, so, ko), 0.30, "1080p L_max=0")
    assert (ko == O.KEEP_NOVELTY).any() and not (ko == O.KEEP_GAP).any()
    f.close()
    # scene changes + H-diff
    two_n = 2 * spec.width * spec.height
    sd = np.array([SC.l1(hist_o[t], hist_o[t - 1]) for t in range(1, spec.frames)]) / two_n
    t_grad, t_cut = float(np.quantile(sd, 0.6)), float(np.quantile(sd, 0.995))
    p3 = O.Params(spec.width, spec.height, tau=0.30, l_max=30)
    so, ko = SC.select(hist_o, p3, t_cut, t_grad)
    assert (ko == SC.KEEP_SCENE).any()
    f = NGFF(spec.width, spec.height, tau=0.30, l_max=30, signal=_abi.SIGNAL_SCD, scd_cut=t_cut, scd_gradual=t_grad,
             max_frames_per_push=spec.frames)
    assert_parity(run_stream(f, dev, [spec.frames]), (hist_o, so, ko), 0.30, "1080p scene changes")
    f.close()
    # scene changes without forced retention (the walk with scanned scene flags)
    so, ko = SC.select(hist_o, O.Params(spec.width, spec.height, tau=0.30, l_max=0), t_cut, t_grad)
    assert (ko == SC.KEEP_SCENE).any() and not (ko == O.KEEP_GAP).any()
    f = NGFF(spec.width, spec.height, tau=0.30, l_max=0, signal=_abi.SIGNAL_SCD, scd_cut=t_cut, scd_gradual=t_grad,
             max_frames_per_push=spec.frames)
    assert_parity(run_stream(f, dev, [spec.frames]), (hist_o, so, ko), 0.30, "1080p scene changes, L_max=0")
    f.close()


def test_rare_event_720p():
    from paper_2609_03675_gb300 import NGFF
    spec = synth.rare_event()
    buf = _pinned_stream(spec)
    dev = buf.cuda()
    taus = (0.30, 0.15, 0.10, 0.05, 0.02)
    hist_o, sel = _oracle(buf, spec, taus)
    events = synth.event_mask(spec).astype(bool)
    for tau in taus:
        f = NGFF(spec.width, spec.height, tau=tau)
        got = run_stream(f, dev, [spec.frames])
        assert_parity(got, (hist_o, *sel[tau]), tau, f"720p tau={tau}")
        kept = got[2] != 0
        print(f"720p tau={tau}: keep ratio {kept.mean():.4f}, event-frame recall {kept[events].mean():.3f}")
        f.close()


def test_serving_32_streams_batched():
    from paper_2609_03675_gb300 import NGFF
    S = synth.SERVING_STREAMS
    specs = [synth.serving_stream(s) for s in range(S)]
    T, W, H = specs[0].frames, specs[0].width, specs[0].height
    o = O.load()
    p = O.Params(W, H)
    host = torch.empty((T, H, W, 3), dtype=torch.uint8, pin_memory=True)
    dev, want = [], []
    for sp in specs:
        synth.generate(sp, out=host.data_ptr())
        hist = o.histograms_parallel(host.data_ptr(), T, p)
        want.append((hist, *o.select(hist, p)))
        dev.append(host.cuda())
    f = NGFF(W, H, max_streams=S)
    sizes = [synth.push_sizes(synth.SEED_BASE + 4, s, T) for s in range(S)]
    scores = torch.empty((S, T), dtype=torch.float32, device="cuda")
    keep = torch.empty((S, T), dtype=torch.uint8, device="cuda")
    pos = [0] * S
    call = 0
    while min(pos) < T:
        items = []
        for s in range(S):
            if pos[s] >= T:
                continue
            n = int(min(sizes[s][call], T - pos[s]))
            items.append((s, dev[s][pos[s]:pos[s] + n], scores[s, pos[s]:pos[s] + n], keep[s, pos[s]:pos[s] + n]))
            pos[s] += n
        f.push_batch(items)
        call += 1
        if call in (1, 2, 57, 201) or min(pos) >= T:  # close every stream at its prefix so far
            for s in range(S):
                got = f.candidates(s).cpu().numpy().astype(np.uint32)
                assert np.array_equal(got, o.candidates(want[s][2][:pos[s]], 4)), f"stream {s} at {pos[s]}"
    torch.cuda.synchronize()
    f.status()
    ks, ss = keep.cpu().numpy(), scores.cpu().numpy()
    for s in range(S):
        _, so, ko = want[s]
        assert np.array_equal(ks[s], ko), f"stream {s}"
        assert (np.abs(ss[s].astype(np.float64) - so) <= 1e-6 * so).all(), f"stream {s}"
    print(f"serving: {call} batched calls, keep ratio {(ks != 0).mean():.4f}")
