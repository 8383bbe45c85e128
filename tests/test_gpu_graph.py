"""Pushes captured into CUDA graphs and replayed.

A push with device frames and outputs may be enqueued while its CUDA stream
captures a graph; every launch of the graph then decides the next frames of
the stream. The decisions of a stream replayed that way, chunk by chunk
from one input buffer, must be the oracle's single-pass result (Sec. 3.2,
Eqs. 2-5), on every selection path (the fused small push, the windowed
distances and scan of larger pushes, batches, L_max = 0) and with ordinary
pushes between the launches. Also the launch chaining those pushes rely on:
frames written by a caller's kernel just before a push."""
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


def _stream(T, w=64, h=48, seed=61, mean=7):
    spec = synth.medium(seed=seed).with_(width=w, height=h, frames=T, mean_scene_len=mean)
    return spec, synth.generate(spec)


def _check(fr, p, scores, keep, hist=None):
    hist_o, so, ko = O.load().run(fr, p)
    assert np.array_equal(keep, ko)
    assert np.all(np.abs(scores.astype(np.float64) - so) <= 1e-6 * so)
    if hist is not None:
        assert np.array_equal(hist.astype(np.uint32), hist_o)


def _capture(fn):
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


@pytest.mark.parametrize("chunk", [8, 100])  # the fused small push; distances + scan + row clearing
def test_captured_push_replays_the_stream(chunk):
    from paper_2609_03675_gb300 import NGFF
    T = 3 * chunk if chunk > 64 else 12 * chunk
    spec, fr = _stream(T)
    p = O.Params(spec.width, spec.height, tau=0.05, l_max=5)
    f = NGFF(spec.width, spec.height, tau=0.05, l_max=5)
    dev = torch.from_numpy(fr).cuda()
    buf = torch.empty_like(dev[:chunk])
    sc = torch.empty(chunk, dtype=torch.float32, device="cuda")
    kp = torch.empty(chunk, dtype=torch.uint8, device="cuda")
    hs = torch.empty((chunk, 32), dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    g = _capture(lambda: f.push(buf, scores=sc, keep=kp, hist=hs))
    assert f.frames_seen() == 0  # nothing ran at capture
    outs = []
    for i in range(0, T, chunk):
        buf.copy_(dev[i:i + chunk])
        g.replay()
        outs.append((sc.clone(), kp.clone(), hs.clone()))
    torch.cuda.synchronize()
    f.status()
    _check(fr, p, torch.cat([o[0] for o in outs]).cpu().numpy(), torch.cat([o[1] for o in outs]).cpu().numpy(),
           torch.cat([o[2] for o in outs]).cpu().numpy())
    assert f.frames_seen() == 0  # graph launches are not counted


def test_captured_and_ordinary_pushes_interleave():
    """Ordinary pushes of both paths between graph launches, on one stream."""
    from paper_2609_03675_gb300 import NGFF
    spec, fr = _stream(500, seed=62)
    p = O.Params(spec.width, spec.height, tau=0.05, l_max=7)
    f = NGFF(spec.width, spec.height, tau=0.05, l_max=7)
    dev = torch.from_numpy(fr).cuda()
    small = torch.empty_like(dev[:9])
    big = torch.empty_like(dev[:90])
    s9 = torch.empty(9, dtype=torch.float32, device="cuda")
    k9 = torch.empty(9, dtype=torch.uint8, device="cuda")
    s90 = torch.empty(90, dtype=torch.float32, device="cuda")
    k90 = torch.empty(90, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    g_small = _capture(lambda: f.push(small, scores=s9, keep=k9))
    g_big = _capture(lambda: f.push(big, scores=s90, keep=k90))
    # (kind, frames): graph launches of both sizes around ordinary pushes of both paths
    plan = [("push", 37), ("big", 90), ("push", 80), ("small", 9), ("small", 9), ("push", 3), ("big", 90),
            ("push", 70), ("big", 90), ("small", 9), ("push", 13)]
    assert sum(n for _, n in plan) == 500
    scores, keep, pos, ordinary = [], [], 0, 0
    for kind, n in plan:
        if kind == "push":
            s, k = f.push(dev[pos:pos + n])
            ordinary += n
        else:
            buf, g, s_out, k_out = (small, g_small, s9, k9) if kind == "small" else (big, g_big, s90, k90)
            buf.copy_(dev[pos:pos + n])
            g.replay()
            s, k = s_out.clone(), k_out.clone()
        scores.append(s)
        keep.append(k)
        pos += n
    torch.cuda.synchronize()
    f.status()
    _check(fr, p, torch.cat(scores).cpu().numpy(), torch.cat(keep).cpu().numpy())
    assert f.frames_seen() == ordinary


def test_captured_batch_of_streams():
    from paper_2609_03675_gb300 import NGFF
    sizes = [5, 8, 3]  # frames per stream per launch
    reps = 14
    streams = [_stream(n * reps, seed=63 + s) for s, n in enumerate(sizes)]
    spec = streams[0][0]
    f = NGFF(spec.width, spec.height, tau=0.05, l_max=6, max_streams=4)
    devs = [torch.from_numpy(fr).cuda() for _, fr in streams]
    bufs = [torch.empty_like(d[:n]) for d, n in zip(devs, sizes)]
    outs = [(torch.empty(n, dtype=torch.float32, device="cuda"), torch.empty(n, dtype=torch.uint8, device="cuda"))
            for n in sizes]
    items = [(s + 1, bufs[s], outs[s][0], outs[s][1]) for s in range(len(sizes))]  # streams 1..3
    arr, nd = f.make_batch(items)
    torch.cuda.synchronize()
    g = _capture(lambda: f.push_batch_raw(arr, nd))
    got = [([], []) for _ in sizes]
    for r in range(reps):
        for s, n in enumerate(sizes):
            bufs[s].copy_(devs[s][r * n:(r + 1) * n])
        g.replay()
        for s in range(len(sizes)):
            got[s][0].append(outs[s][0].clone())
            got[s][1].append(outs[s][1].clone())
    torch.cuda.synchronize()
    f.status()
    for s, (sp, fr) in enumerate(streams):
        _check(fr, O.Params(sp.width, sp.height, tau=0.05, l_max=6), torch.cat(got[s][0]).cpu().numpy(),
               torch.cat(got[s][1]).cpu().numpy())


def test_captured_push_without_forced_retention():
    from paper_2609_03675_gb300 import NGFF
    chunk, T = 16, 160
    spec, fr = _stream(T, seed=66)
    f = NGFF(spec.width, spec.height, tau=0.04, l_max=0)
    dev = torch.from_numpy(fr).cuda()
    buf = torch.empty_like(dev[:chunk])
    sc = torch.empty(chunk, dtype=torch.float32, device="cuda")
    kp = torch.empty(chunk, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    g = _capture(lambda: f.push(buf, scores=sc, keep=kp))
    s_all, k_all = [], []
    for i in range(0, T, chunk):
        buf.copy_(dev[i:i + chunk])
        g.replay()
        s_all.append(sc.clone())
        k_all.append(kp.clone())
    torch.cuda.synchronize()
    f.status()
    _check(fr, O.Params(spec.width, spec.height, tau=0.04, l_max=0), torch.cat(s_all).cpu().numpy(),
           torch.cat(k_all).cpu().numpy())


def test_capture_refuses_host_memory():
    """Host frames or outputs while capturing are argument errors found before
    anything is enqueued: the capture stays valid and its other pushes run."""
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    spec, fr = _stream(24, seed=67)
    f = NGFF(spec.width, spec.height, tau=0.05)
    dev = torch.from_numpy(fr).cuda()
    host = torch.from_numpy(fr[:8].copy())
    sc = torch.empty(8, dtype=torch.float32, device="cuda")
    kp = torch.empty(8, dtype=torch.uint8, device="cuda")
    sc_host = torch.empty(8, dtype=torch.float32)
    buf = torch.empty_like(dev[:8])
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        with pytest.raises(NGFFError) as e1:
            f.push(host, scores=sc, keep=kp)
        with pytest.raises(NGFFError) as e2:
            f.push(buf, scores=sc_host, keep=kp)
        with pytest.raises(NGFFError) as e3:  # the batched call: host frames
            f.push_batch([(0, host, sc, kp)])
        with pytest.raises(NGFFError) as e4:  # and host outputs
            f.push_batch([(0, buf, sc_host, kp)])
        f.push(buf, scores=sc, keep=kp)
    assert all(e.value.code == _abi.EINVAL for e in (e1, e2, e3, e4))
    assert "device frames and outputs only" in str(e3.value) and "device frames and outputs only" in str(e4.value)
    s_all, k_all = [], []
    for i in range(0, 24, 8):
        buf.copy_(dev[i:i + 8])
        g.replay()
        s_all.append(sc.clone())
        k_all.append(kp.clone())
    torch.cuda.synchronize()
    f.status()
    _check(fr, O.Params(spec.width, spec.height, tau=0.05), torch.cat(s_all).cpu().numpy(),
           torch.cat(k_all).cpu().numpy())


@pytest.mark.parametrize("chunk", [8, 100])
def test_frames_written_by_a_kernel_just_before_each_push(chunk):
    """The first-stage kernel is a programmatic dependent of the kernel before
    it; when that kernel is the caller's and writes the frames, the push must
    still read them complete. Each chunk is decoded (an elementwise XOR
    kernel) into the input buffer immediately before its push, with no other
    work between."""
    from paper_2609_03675_gb300 import NGFF
    T = 400
    spec, fr = _stream(T, seed=68)
    p = O.Params(spec.width, spec.height, tau=0.05, l_max=9)
    f = NGFF(spec.width, spec.height, tau=0.05, l_max=9)
    dev = torch.from_numpy(fr).cuda()
    gen = torch.Generator(device="cuda").manual_seed(5)
    noise = torch.randint(0, 256, dev.shape, dtype=torch.uint8, device="cuda", generator=gen)
    enc = torch.bitwise_xor(dev, noise)
    del dev
    buf = torch.empty_like(enc[:chunk])
    scores, keep = [], []
    for i in range(0, T, chunk):
        n = min(chunk, T - i)
        torch.bitwise_xor(enc[i:i + n], noise[i:i + n], out=buf[:n])
        s, k = f.push(buf[:n])
        scores.append(s)
        keep.append(k)
    torch.cuda.synchronize()
    f.status()
    _check(fr, p, torch.cat(scores).cpu().numpy(), torch.cat(keep).cpu().numpy())


@pytest.mark.parametrize("signal", ["lowres", "dhash"])
@pytest.mark.parametrize("chunk", [8, 100])
def test_captured_push_spatial_signals(signal, chunk):
    """The ablation's signals under capture: low-res cell sums (rows cleared
    after use like histograms) and dHash (cell sums cleared by the hash
    kernel, hash rows written whole), replayed chunk by chunk."""
    from oracle import signals_oracle as SO
    from paper_2609_03675_gb300 import NGFF, _abi
    from tests.test_gpu_signals import _tau_for
    kind = SO.LOWRES if signal == "lowres" else SO.DHASH
    T, W, H = 3 * chunk if chunk > 64 else 12 * chunk, 160, 90
    spec, fr = _stream(T, w=W, h=H, seed=69)
    feats = np.stack([SO.features(x, O.Params(W, H), kind) for x in fr])
    tau = _tau_for(feats, O.Params(W, H), kind, l_max=6)
    p = O.Params(W, H, tau=tau, l_max=6)
    so, ko = SO.select(feats, p, kind)
    assert (ko == O.KEEP_NOVELTY).any() and (ko == O.KEEP_DROP).any()
    sig = _abi.SIGNAL_LOWRES if signal == "lowres" else _abi.SIGNAL_DHASH
    f = NGFF(W, H, tau=tau, l_max=6, signal=sig)
    dev = torch.from_numpy(fr).cuda()
    buf = torch.empty_like(dev[:chunk])
    sc = torch.empty(chunk, dtype=torch.float32, device="cuda")
    kp = torch.empty(chunk, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    g = _capture(lambda: f.push(buf, scores=sc, keep=kp))
    s_all, k_all = [], []
    for i in range(0, T, chunk):
        buf.copy_(dev[i:i + chunk])
        g.replay()
        s_all.append(sc.clone())
        k_all.append(kp.clone())
    torch.cuda.synchronize()
    f.status()
    kg = torch.cat(k_all).cpu().numpy()
    sg = torch.cat(s_all).cpu().numpy().astype(np.float64)
    assert np.array_equal(kg, ko)
    assert np.all(np.abs(sg - so) <= 1e-6 * so)
