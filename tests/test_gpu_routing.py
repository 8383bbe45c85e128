"""The first stage runs either the bulk-copy histogram kernel (K1) or the
generic one, chosen per launch by its size: the generic kernel when its grid
(one CTA per 2048 16-pixel groups of a frame) holds at least two CTAs per SM
and fits one resident wave plus an eighth. Pushes sized just below, at and
above those boundaries, plain and with histograms out, one stream and
batched, give the oracle's histograms, scores and keep codes whichever
kernel ran."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.gpu_helpers import assert_parity, oracle_run, run_stream

pytestmark = pytest.mark.gpu

W, H = 64, 48  # 192 groups: one generic CTA per frame, so a push of n frames is n generic CTAs


@pytest.fixture(scope="module")
def n_sms():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.cuda.get_device_properties(0).multi_processor_count


def _sizes(n):
    # below and at 2 CTAs per SM; one wave at 6, 7 and 8 CTAs per SM; an eighth past 8; beyond
    return [2 * n - 1, 2 * n, 6 * n, 7 * n, 8 * n, 9 * n, 9 * n + 1, 11 * n]


@pytest.mark.parametrize("bins,l_max,tau", [(32, 30, 0.05), (7, 33, 0.10), (256, 5, 0.02), (1, 1, 0.30)])
def test_pushes_across_the_first_stage_boundaries(n_sms, bins, l_max, tau):
    from paper_2609_03675_gb300 import NGFF
    sizes = _sizes(n_sms)
    T = sum(sizes)
    spec = synth.medium(seed=77).with_(width=W, height=H, frames=T, mean_scene_len=15)
    fr = synth.generate(spec)
    want = oracle_run(fr, O.Params(W, H, bins=bins, l_max=l_max, tau=tau))
    dev = torch.from_numpy(fr).cuda()
    f = NGFF(W, H, bins=bins, l_max=l_max, tau=tau, max_frames_per_push=max(sizes))
    assert_parity(run_stream(f, dev, sizes), want, tau, f"B={bins} L={l_max} with histograms")
    # the same pieces without histograms out (the selection kernels then clear the rows)
    g = NGFF(W, H, bins=bins, l_max=l_max, tau=tau, max_frames_per_push=max(sizes))
    off, ss, ks = 0, [], []
    for n in sizes:
        s, k = g.push(dev[off:off + n])
        ss.append(s)
        ks.append(k)
        off += n
    torch.cuda.synchronize()
    g.status()
    _, so, ko = want
    kg = torch.cat(ks).cpu().numpy()
    sg = torch.cat(ss).cpu().numpy().astype(np.float64)
    assert np.array_equal(kg, ko), np.flatnonzero(kg != ko)[:10]
    assert np.all(np.abs(sg - so) <= 1e-6 * so)
    f.close()
    g.close()


def test_batched_calls_across_the_boundaries(n_sms):
    """Two streams per batched call whose combined frame count falls below,
    inside and above the generic kernel's window."""
    from paper_2609_03675_gb300 import NGFF
    per_call = [(n_sms - 1, n_sms - 1), (n_sms, n_sms), (3 * n_sms, 3 * n_sms), (4 * n_sms, 5 * n_sms),
                (5 * n_sms, 5 * n_sms), (1, 2 * n_sms)]
    T = [sum(c[s] for c in per_call) for s in range(2)]
    specs = [synth.medium(seed=90 + s).with_(width=W, height=H, frames=T[s], mean_scene_len=12) for s in range(2)]
    frs = [synth.generate(sp) for sp in specs]
    wants = [oracle_run(x, O.Params(W, H, tau=0.05)) for x in frs]
    devs = [torch.from_numpy(x).cuda() for x in frs]
    outs = [(torch.empty(t, dtype=torch.float32, device="cuda"), torch.empty(t, dtype=torch.uint8, device="cuda"))
            for t in T]
    f = NGFF(W, H, tau=0.05, max_streams=2, max_frames_per_push=16 * n_sms)
    pos = [0, 0]
    for c in per_call:
        items = []
        for s in range(2):
            a, n = pos[s], c[s]
            items.append((s, devs[s][a:a + n], outs[s][0][a:a + n], outs[s][1][a:a + n]))
            pos[s] += n
        f.push_batch(items)
    torch.cuda.synchronize()
    f.status()
    for s in range(2):
        _, so, ko = wants[s]
        kg = outs[s][1].cpu().numpy()
        assert np.array_equal(kg, ko), (s, np.flatnonzero(kg != ko)[:10])
        assert np.all(np.abs(outs[s][0].cpu().numpy().astype(np.float64) - so) <= 1e-6 * so)
    f.close()
