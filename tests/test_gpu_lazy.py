"""L_max = 0 (no forced retention; Eq. 5's second term off): the rule walked
in frame order by one warp per stream, against the oracles (C for the
histogram, Python for the other signals) read the same way."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from oracle import scd_oracle as SC
from oracle import signals_oracle as SO

from tests.gpu_helpers import SCORE_RTOL, assert_parity, run_stream

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _frames(w, h, T, seed, mean=9):
    return synth.generate(synth.medium(seed=seed).with_(width=w, height=h, frames=T, mean_scene_len=mean))


@pytest.mark.parametrize("bins,tau", [(32, 0.05), (32, 0.3), (7, 0.08), (256, 0.1), (1, 0.0), (32, 1.5)])
def test_histogram_rule_without_gap(bins, tau):
    from paper_2609_03675_gb300 import NGFF
    w, h, T = 64, 48, 700
    fr = _frames(w, h, T, seed=700 + bins)
    p = O.Params(w, h, bins=bins, tau=tau, l_max=0)
    want = O.load().run(fr, p)
    assert not (want[2] == O.KEEP_GAP).any()
    dev = torch.from_numpy(fr).cuda()
    for chunks in ([T], [1, 2, 63, 64, 65, 505], [1] * 40 + [T - 40]):
        f = NGFF(w, h, bins=bins, tau=tau, l_max=0, max_frames_per_push=1024)
        assert_parity(run_stream(f, dev, chunks), want, tau, f"bins {bins} chunks {chunks[:3]}")


def test_long_stream_many_tiles_and_host_frames():
    from paper_2609_03675_gb300 import NGFF
    w, h, T = 32, 24, 9000  # several 256-row shared-memory tiles per push
    fr = _frames(w, h, T, seed=711, mean=40)
    p = O.Params(w, h, tau=0.04, l_max=0)
    _, so, ko = O.load().run(fr, p)
    f = NGFF(w, h, tau=0.04, l_max=0, max_frames_per_push=T)
    s, k = f.push(torch.from_numpy(fr).pin_memory())  # host frames and outputs
    torch.cuda.synchronize()
    f.status()
    assert np.array_equal(k.numpy(), ko)
    assert (np.abs(s.numpy().astype(np.float64) - so) <= SCORE_RTOL * so).all()
    assert (ko != 0).sum() > 50 and (ko == 0).sum() > 50


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_spatial_signals_without_gap(kind):
    from paper_2609_03675_gb300 import NGFF
    w, h, T = 64, 48, 300
    fr = _frames(w, h, T, seed=720 + kind)
    tau = 0.03 if kind == SO.LOWRES else 0.1
    _, so, ko = SO.run(fr, O.Params(w, h, tau=tau, l_max=0), kind)
    f = NGFF(w, h, tau=tau, l_max=0, signal=kind)
    _, sg, kg = run_stream(f, torch.from_numpy(fr).cuda(), [100, 1, 199])
    assert np.array_equal(kg, ko)
    assert (np.abs(sg.astype(np.float64) - so) <= SCORE_RTOL * so).all()


def test_scene_change_signal_without_gap_and_state():
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    w, h, T = 64, 48, 400
    fr = _frames(w, h, T, seed=731, mean=15)
    p = O.Params(w, h, tau=0.35, l_max=0)
    hist = np.stack([O.load().histogram(x, p) for x in fr])
    sd = np.array([SC.l1(hist[t], hist[t - 1]) for t in range(1, T)]) / (2 * w * h)
    t_grad, t_cut = float(np.quantile(sd, 0.5)), float(np.quantile(sd, 0.97))
    so, ko = SC.select(hist, p, t_cut, t_grad)
    assert (ko == SC.KEEP_SCENE).any()
    dev = torch.from_numpy(fr).cuda()
    kw = dict(tau=0.35, l_max=0, signal=_abi.SIGNAL_SCD, scd_cut=t_cut, scd_gradual=t_grad)
    a = NGFF(w, h, **kw)
    s1, k1 = a.push(dev[:173])
    state = a.state_save()
    b = NGFF(w, h, **kw)
    b.state_load(state)
    s2, k2 = b.push(dev[173:])
    torch.cuda.synchronize()
    b.status()
    assert np.array_equal(torch.cat([k1, k2]).cpu().numpy(), ko)
    assert (np.abs(torch.cat([s1, s2]).cpu().numpy().astype(np.float64) - so) <= SCORE_RTOL * so).all()
    with pytest.raises(NGFFError) as e:
        NGFF(w, h, tau=0.35, l_max=0).shard_prepare(dev[:10], n_halo=0, t0=0)
    assert e.value.code == _abi.EINVAL


def test_batch_of_streams_without_gap():
    from paper_2609_03675_gb300 import NGFF
    w, h, S, T = 48, 32, 6, 120
    frs = [_frames(w, h, T, seed=740 + s, mean=6) for s in range(S)]
    f = NGFF(w, h, tau=0.06, l_max=0, max_streams=S)
    dev = [torch.from_numpy(x).cuda() for x in frs]
    outs = {s: [] for s in range(S)}
    for a, b in ((0, 50), (50, 51), (51, 120)):
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
        _, so, ko = O.load().run(frs[s], O.Params(w, h, tau=0.06, l_max=0))
        assert np.array_equal(torch.cat([k for _, k in outs[s]]).cpu().numpy(), ko), f"stream {s}"
