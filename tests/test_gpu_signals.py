"""The alternative pre-encoder signals (low-res difference, dHash) against
their oracle: each replaces the histogram distance in the same retention rule
(Sec. 3.2, Eqs. 3-5; the signal ablation table). Per-frame features are
compared bit for bit, scores within the fp32 rounding bound, keep codes
exactly (both sides decide fp32(numerator) / fp32(denominator) >= tau)."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from oracle import signals_oracle as SO

from tests.gpu_helpers import SCORE_RTOL, run_stream

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _frames(w, h, T, seed, mean=8):
    spec = synth.medium(seed=seed).with_(width=w, height=h, frames=T, mean_scene_len=mean)
    return synth.generate(spec)


def _unpack(words: np.ndarray) -> np.ndarray:
    """dHash words [T, 2] -> bits [T, 64], bit i = bit (i % 32) of word i // 32."""
    w = words.astype(np.uint64)
    return np.concatenate([(w[:, [k]] >> np.arange(32, dtype=np.uint64)) & 1 for k in range(2)], axis=1)


def _tau_for(feats, p, kind, l_max=30):
    """A threshold inside the distribution of adjacent distances at which the
    rule both keeps frames for novelty and drops others (the oracle decides)."""
    den = SO.denominator(p, kind)
    adj = np.array([SO.numerator(feats[t], feats[t - 1], kind) / den for t in range(1, len(feats))])
    pos = adj[adj > 0]
    for q in (0.7, 0.5, 0.85, 0.3, 0.95):
        tau = float(np.float32(max(np.quantile(adj, q), pos.min() if pos.size else 1.0)))
        _, ko = SO.select(feats, O.Params(p.width, p.height, tau=tau, l_max=l_max, luma_w=p.luma_w,
                                          luma_den=p.luma_den), kind)
        if (ko == O.KEEP_NOVELTY).any() and (ko == O.KEEP_DROP).any():
            return tau
    return tau


def _check(f, fr, kind, l_max, chunks, label):
    H, W = fr.shape[1:3]
    feats = np.stack([SO.features(x, O.Params(W, H), kind) for x in fr])
    tau = _tau_for(feats, O.Params(W, H), kind, l_max)
    p = O.Params(W, H, tau=tau, l_max=l_max)
    so, ko = SO.select(feats, p, kind)
    assert (ko == O.KEEP_NOVELTY).any() and (ko == O.KEEP_DROP).any(), "workload exercises both outcomes"
    g = f(tau)
    hg, sg, kg = run_stream(g, torch.from_numpy(fr).cuda(), chunks)
    got = hg.astype(np.int64) if kind == SO.LOWRES else _unpack(hg)
    bad = np.flatnonzero((got != feats).any(axis=1))
    assert len(bad) == 0, f"{label}: features differ at frames {list(bad[:10])}"
    err = np.abs(sg.astype(np.float64) - so)
    assert (err <= SCORE_RTOL * so).all(), f"{label}: scores differ at {list(np.flatnonzero(err > SCORE_RTOL * so)[:10])}"
    badkeep = np.flatnonzero(kg != ko)
    assert len(badkeep) == 0, f"{label}: keep codes differ at {list(badkeep[:10])}"


SHAPES = [
    (64, 48),    # width % 16 == 0: 16-pixel vector path
    (72, 40),    # width % 16 == 8: byte path
    (37, 23),    # odd sizes, uneven cells
    (16, 16),    # one pixel per low-res cell
    (160, 90),   # dHash cells wider than a 16-pixel group
    (272, 20),   # both signals: cells of 17 and 30 pixels, uneven rows
]


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
@pytest.mark.parametrize("shape", SHAPES)
def test_signal_matches_oracle(kind, shape):
    from paper_2609_03675_gb300 import NGFF
    W, H = shape
    T = 260
    fr = _frames(W, H, T, seed=900 + W + kind)
    for l_max, chunks in ((30, [T]), (7, [1, 2, 61, 64, 132]), (256, [100, 160])):
        _check(lambda tau: NGFF(W, H, tau=tau, l_max=l_max, signal=kind), fr, kind, l_max, chunks,
               f"{W}x{H} kind {kind} L {l_max} chunks {chunks}")


def test_dhash_smallest_frame():
    from paper_2609_03675_gb300 import NGFF
    fr = _frames(9, 8, 120, seed=931)
    _check(lambda tau: NGFF(9, 8, tau=tau, l_max=5, signal=SO.DHASH), fr, SO.DHASH, 5, [50, 70], "9x8")


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_signal_1080p_sampled(kind):
    """Full-size frames: a short stream decided whole by the oracle."""
    from paper_2609_03675_gb300 import NGFF
    spec = synth.hd1080()
    fr = synth.generate(spec, 0, 48)
    W, H = spec.width, spec.height
    _check(lambda tau: NGFF(W, H, tau=tau, signal=kind, max_frames_per_push=64), fr, kind, 30, [3, 45],
           f"1080p kind {kind}")


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_signal_batch_of_streams(kind):
    from paper_2609_03675_gb300 import NGFF
    W, H, S, T = 64, 48, 5, 90
    tau = 0.04 if kind == SO.LOWRES else 0.12
    fr = [_frames(W, H, T, seed=950 + s) for s in range(S)]
    f = NGFF(W, H, tau=tau, l_max=11, signal=kind, max_streams=S)
    dev = [torch.from_numpy(x).cuda() for x in fr]
    outs = {s: [] for s in range(S)}
    for a, b in ((0, 40), (40, 41), (41, 90)):
        items = []
        for s in range(S):
            sc = torch.empty(b - a, dtype=torch.float32, device="cuda")
            kp = torch.empty(b - a, dtype=torch.uint8, device="cuda")
            items.append((s, dev[s][a:b], sc, kp))
            outs[s].append((sc, kp))
        f.push_batch(items)
    torch.cuda.synchronize()
    f.status()
    for s in range(S):
        _, so, ko = SO.run(fr[s], O.Params(W, H, tau=tau, l_max=11), kind)
        kg = torch.cat([k for _, k in outs[s]]).cpu().numpy()
        sg = torch.cat([x for x, _ in outs[s]]).cpu().numpy().astype(np.float64)
        assert np.array_equal(kg, ko), f"stream {s}"
        assert (np.abs(sg - so) <= SCORE_RTOL * so).all(), f"stream {s}"


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_signal_state_and_shards(kind):
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    W, H, T, L = 64, 48, 200, 9
    tau = 0.04 if kind == SO.LOWRES else 0.12
    fr = _frames(W, H, T, seed=970 + kind)
    _, so, ko = SO.run(fr, O.Params(W, H, tau=tau, l_max=L), kind)
    dev = torch.from_numpy(fr).cuda()
    # checkpoint and resume on another handle
    a = NGFF(W, H, tau=tau, l_max=L, signal=kind)
    s1, k1 = a.push(dev[:77])
    state = a.state_save()
    b = NGFF(W, H, tau=tau, l_max=L, signal=kind)
    b.state_load(state)
    s2, k2 = b.push(dev[77:])
    torch.cuda.synchronize()
    assert np.array_equal(torch.cat([k1, k2]).cpu().numpy(), ko)
    assert (np.abs(torch.cat([s1, s2]).cpu().numpy().astype(np.float64) - so) <= SCORE_RTOL * so).all()
    other = SO.DHASH if kind == SO.LOWRES else 0
    with pytest.raises(NGFFError) as e:
        NGFF(W, H, tau=tau, l_max=L, signal=other).state_load(state)
    assert e.value.code == _abi.EINVAL
    # two shards prepared in reverse order and chained through the gap map
    cut = 120
    second = NGFF(W, H, tau=tau, l_max=L, signal=kind)
    m = second.shard_prepare(dev[cut - L:], n_halo=L, t0=cut).numpy()
    first = NGFF(W, H, tau=tau, l_max=L, signal=kind)
    m1 = first.shard_prepare(dev[:cut], n_halo=0, t0=0).numpy()
    sa, ka = first.shard_commit(1, cut)
    torch.cuda.synchronize()
    g_exit = int(m1[0])
    assert g_exit == cut - np.flatnonzero(ka.cpu().numpy())[-1], "exit gap is t - r(t) past the shard's end"
    sb, kb = second.shard_commit(g_exit, T - cut)
    torch.cuda.synchronize()
    assert np.array_equal(torch.cat([ka, kb]).cpu().numpy(), ko)
    assert (np.abs(torch.cat([sa, sb]).cpu().numpy().astype(np.float64) - so) <= SCORE_RTOL * so).all()
    assert m.shape[0] == L


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_signal_unaligned_frames_and_plain_division(kind):
    """Frames at an odd address (the per-frame byte path) and a grayscale
    divisor of 1 (no multiply-high: the per-frame kernel's 16-pixel path)."""
    from paper_2609_03675_gb300 import NGFF
    W, H, T = 64, 48, 150
    fr = _frames(W, H, T, seed=990 + kind)
    raw = torch.empty(fr.size + 1, dtype=torch.uint8, device="cuda")
    raw[1:].copy_(torch.from_numpy(fr.reshape(-1)))
    odd = raw[1:].view(T, H, W, 3)
    feats = np.stack([SO.features(x, O.Params(W, H), kind) for x in fr])
    tau = _tau_for(feats, O.Params(W, H), kind, 13)
    _, so, ko = SO.run(fr, O.Params(W, H, tau=tau, l_max=13), kind)
    g = NGFF(W, H, tau=tau, l_max=13, signal=kind)
    s, k = g.push(odd)
    torch.cuda.synchronize()
    g.status()
    assert np.array_equal(k.cpu().numpy(), ko)
    assert (np.abs(s.cpu().numpy().astype(np.float64) - so) <= SCORE_RTOL * so).all()
    # grayscale = R (weights 1, 0, 0 over 1)
    pr = O.Params(W, H, luma_w=(1, 0, 0), luma_den=1)
    feats = np.stack([SO.features(x, pr, kind) for x in fr])
    tau = _tau_for(feats, pr, kind, 13)
    _, so, ko = SO.run(fr, O.Params(W, H, tau=tau, l_max=13, luma_w=(1, 0, 0), luma_den=1), kind)
    g = NGFF(W, H, tau=tau, l_max=13, signal=kind, luma_weights=(1, 0, 0), luma_den=1)
    s, k, f = g.push(torch.from_numpy(fr).cuda(), return_hist=True)
    torch.cuda.synchronize()
    g.status()
    got = f.cpu().numpy().view(np.uint32)
    got = got.astype(np.int64) if kind == SO.LOWRES else _unpack(got)
    assert np.array_equal(got, feats)
    assert np.array_equal(k.cpu().numpy(), ko)
    assert (np.abs(s.cpu().numpy().astype(np.float64) - so) <= SCORE_RTOL * so).all()
