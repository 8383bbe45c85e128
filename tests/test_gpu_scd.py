"""Scene change detection + H-diff on the GPU against its oracle: twin
comparison of adjacent histogram differences added to the histogram rule
(the signal ablation, Table "hdiff-signal"; readings in the oracle's header).
Keep codes must be identical, scores within the fp32 rounding bound."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from oracle import scd_oracle as SC

from tests.gpu_helpers import SCORE_RTOL

pytestmark = pytest.mark.gpu

W = H = 32
N = W * H


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _frames_from_positions(pos):
    """Frame t: its first pos[t] pixels (row-major) white, the rest black; the
    B-bin histogram then has pos[t] counts in the top bin and N - pos[t] in bin 0."""
    pos = np.asarray(pos)
    fr = np.zeros((len(pos), N, 3), dtype=np.uint8)
    fr[np.arange(N)[None, :] < pos[:, None]] = 255
    return fr.reshape(len(pos), H, W, 3)


def _walk(T, seed):
    """Bin-top counts of a random walk: holds, low steps (4 px, SD = 1/256),
    middle steps (16 px, SD = 1/64) in runs, and cuts (300 px)."""
    g = np.random.default_rng(seed)
    pos, p = [], 512
    while len(pos) < T:
        kind = g.choice(4, p=[0.25, 0.2, 0.5, 0.05])
        n = int(g.integers(1, 14)) if kind == 2 else 1
        step = (0, 4, 16, 300)[kind] * (1 if g.random() < 0.5 else -1)
        for _ in range(n):
            if not 0 <= p + step <= N:
                step = -step
            p += step
            pos.append(p)
    return pos[:T]


def _run(f, dev, chunks):
    ss, ks = [], []
    off = 0
    for c in chunks:
        s, k = f.push(dev[off:off + c])
        ss.append(s)
        ks.append(k)
        off += c
    torch.cuda.synchronize()
    f.status()
    return torch.cat(ss).cpu().numpy().astype(np.float64), torch.cat(ks).cpu().numpy()


def _oracle(fr, p, t_cut, t_grad):
    hist = np.stack([O.load().histogram(x, p) for x in fr])
    return SC.select(hist, p, t_cut, t_grad)


def _assert_same(sg, kg, so, ko, label=""):
    bad = np.flatnonzero(kg != ko)
    assert len(bad) == 0, f"{label}: keep codes differ at {list(bad[:10])}: {kg[bad[:5]]} vs {ko[bad[:5]]}"
    err = np.abs(sg - so)
    assert (err <= SCORE_RTOL * so).all(), f"{label}: scores differ at {list(np.flatnonzero(err > SCORE_RTOL * so)[:5])}"


def test_two_ramps_closed_form_on_device():
    """The oracle's hand-derived case (scene changes at 8 and 31, novelty at 63)
    realised as frames, pushed whole and frame by frame."""
    from paper_2609_03675_gb300 import NGFF, _abi
    pos = [16 * t for t in range(21)] + [320] * 3 + [320 + 16 * (t - 23) for t in range(24, 64)]
    dev = torch.from_numpy(_frames_from_positions(pos)).cuda()
    for l_max in (256, 0):  # the window + scan kernels, and the frame-order walk
        for chunks in ([64], [1] * 64, [5, 30, 29]):
            f = NGFF(W, H, tau=0.5, l_max=l_max, signal=_abi.SIGNAL_SCD, scd_cut=0.125, scd_gradual=0.01)
            _, k = _run(f, dev, chunks)
            assert {int(t): int(k[t]) for t in np.flatnonzero(k)} == {0: 3, 8: 4, 31: 4, 63: 1}, (l_max, chunks)


@pytest.mark.parametrize("tau,l_max", [(0.5, 30), (1.5, 7), (0.2, 256), (0.5, 0)])
def test_random_walk_long_stream(tau, l_max):
    """12,000 frames: several 4096-frame scan tiles, runs crossing tile and
    push boundaries, pushes through both the fused small-push kernel and the
    window + scan kernels."""
    from paper_2609_03675_gb300 import NGFF, _abi
    T = 12000
    pos = _walk(T, seed=int(tau * 100) + l_max)
    fr = _frames_from_positions(pos)
    p = O.Params(W, H, tau=tau, l_max=l_max)
    so, ko = _oracle(fr, p, 0.125, 0.01)
    assert (ko == SC.KEEP_SCENE).sum() > 20
    dev = torch.from_numpy(fr).cuda()
    for chunks in ([T], [1, 63, 64, 4000, 4097, 10, T - 8235], [37] * (T // 37) + [T % 37]):
        f = NGFF(W, H, tau=tau, l_max=l_max, signal=_abi.SIGNAL_SCD, scd_cut=0.125, scd_gradual=0.01,
                 max_frames_per_push=T)
        sg, kg = _run(f, dev, chunks)
        _assert_same(sg, kg, so, ko, f"chunks {chunks[:4]}")


def test_synthetic_scenes_and_batches():
    """Seeded scene streams (cuts, drift, noise) with thresholds inside their
    adjacent-difference distribution, five streams through one batched call."""
    from paper_2609_03675_gb300 import NGFF, _abi
    S, T, w, h = 5, 400, 64, 48
    frs = [synth.generate(synth.medium(seed=300 + s).with_(width=w, height=h, frames=T, mean_scene_len=12))
           for s in range(S)]
    p0 = O.Params(w, h)
    hist0 = np.stack([O.load().histogram(x, p0) for x in frs[0]])
    sd = np.array([SC.l1(hist0[t], hist0[t - 1]) for t in range(1, T)]) / (2 * w * h)
    t_grad, t_cut = float(np.quantile(sd, 0.5)), float(np.quantile(sd, 0.97))
    p = O.Params(w, h, tau=0.3, l_max=20)
    f = NGFF(w, h, tau=0.3, l_max=20, signal=_abi.SIGNAL_SCD, scd_cut=t_cut, scd_gradual=t_grad, max_streams=S)
    dev = [torch.from_numpy(x).cuda() for x in frs]
    outs = {s: [] for s in range(S)}
    for a, b in ((0, 150), (150, 151), (151, 400)):
        items = []
        for s in range(S):
            sc = torch.empty(b - a, dtype=torch.float32, device="cuda")
            kp = torch.empty(b - a, dtype=torch.uint8, device="cuda")
            items.append((s, dev[s][a:b], sc, kp))
            outs[s].append((sc, kp))
        f.push_batch(items)
    torch.cuda.synchronize()
    f.status()
    scenes = 0
    for s in range(S):
        so, ko = _oracle(frs[s], p, t_cut, t_grad)
        scenes += int((ko == SC.KEEP_SCENE).sum())
        kg = torch.cat([k for _, k in outs[s]]).cpu().numpy()
        sg = torch.cat([x for x, _ in outs[s]]).cpu().numpy().astype(np.float64)
        _assert_same(sg, kg, so, ko, f"stream {s}")
    assert scenes > 0


def test_state_carries_an_open_run_and_sharding_is_refused():
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    pos = [16 * t for t in range(40)]  # one long run: scene change at t = 8, then none
    fr = _frames_from_positions(pos)
    p = O.Params(W, H, tau=1.5, l_max=256)
    so, ko = _oracle(fr, p, 0.125, 0.01)
    dev = torch.from_numpy(fr).cuda()
    kw = dict(tau=1.5, l_max=256, signal=_abi.SIGNAL_SCD, scd_cut=0.125, scd_gradual=0.01)
    for cut in (5, 8, 9, 20):  # save inside the run, before and after its detection
        a = NGFF(W, H, **kw)
        s1, k1 = a.push(dev[:cut])
        state = a.state_save()
        b = NGFF(W, H, **kw)
        b.state_load(state)
        s2, k2 = b.push(dev[cut:])
        torch.cuda.synchronize()
        b.status()
        _assert_same(torch.cat([s1, s2]).cpu().numpy().astype(np.float64), torch.cat([k1, k2]).cpu().numpy(),
                     so, ko, f"cut {cut}")
    with pytest.raises(NGFFError) as e:
        NGFF(W, H, **kw).shard_prepare(dev[:10], n_halo=0, t0=0)
    assert e.value.code == _abi.EINVAL
    with pytest.raises(NGFFError):  # a histogram-signal state does not load into a scene-change handle
        NGFF(W, H, **kw).state_load(NGFF(W, H, tau=1.5, l_max=256).state_save())


@pytest.mark.parametrize("t_cut,t_grad", [(0.02, 0.05), (0.03, 0.03)])
@pytest.mark.parametrize("l_max", [30, 0])
def test_gradual_threshold_at_or_above_the_cut(t_cut, t_grad, l_max):
    """T_s >= T_b: no difference lies between them, so no run ever opens and
    every scene change is a cut; both selection kernels (scan tiles for
    L_max > 0, the walk with scanned scene flags for L_max = 0) must agree
    with the oracle."""
    from paper_2609_03675_gb300 import NGFF, _abi
    T = 3000
    pos = _walk(T, seed=900 + l_max)
    fr = _frames_from_positions(pos)
    p = O.Params(W, H, tau=1.5, l_max=l_max)
    so, ko = _oracle(fr, p, t_cut, t_grad)
    assert (ko == SC.KEEP_SCENE).sum() > 10
    dev = torch.from_numpy(fr).cuda()
    for chunks in ([T], [1, 999, 2000]):
        f = NGFF(W, H, tau=1.5, l_max=l_max, signal=_abi.SIGNAL_SCD, scd_cut=t_cut, scd_gradual=t_grad,
                 max_frames_per_push=T)
        sg, kg = _run(f, dev, chunks)
        _assert_same(sg, kg, so, ko, f"T_b {t_cut} T_s {t_grad} L_max {l_max} {chunks[:2]}")
