"""Frames at the largest sizes the ABI accepts, where every 32-bit count,
index and L1 numerator is closest to its limit: W·H just under 2^31 pixels
(6.4 GB per frame; a histogram bin can hold every pixel and the L1 numerator
2N stays below 2^32) on the fast kernel (W·H a multiple of 16) and on the
generic one, and the low-res signal at its own limit of 2^24 pixels."""
import gc

import numpy as np
import pytest
import torch

import oracle as O
import synth
from oracle import signals_oracle as SO

from tests.gpu_helpers import SCORE_RTOL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _frames(w, h, T, seed):
    spec = synth.hd1080(seed=seed).with_(width=w, height=h, frames=T)
    return synth.generate(spec)


def _limit_frames(w, h, seed):
    """Three frames of w x h: a seeded random 1 MiB block repeated over the
    frame (every bin populated), then all black (bin 0 holds every pixel),
    then all white (the L1 numerator to the black frame is 2N)."""
    fb = 3 * w * h
    g = np.random.default_rng(seed)
    block = g.integers(0, 256, size=3 * 349525, dtype=np.uint8)
    fr = np.empty((3, fb), dtype=np.uint8)
    reps = fb // block.size
    fr[0, : reps * block.size].reshape(reps, block.size)[:] = block
    fr[0, reps * block.size:] = block[: fb - reps * block.size]
    fr[1] = 0
    fr[2] = 255
    return fr.reshape(3, h, w, 3)


@pytest.mark.parametrize("w,h", [(46336, 46336), (46339, 46342)])
def test_histogram_at_the_pixel_limit(w, h):
    from paper_2609_03675_gb300 import NGFF
    assert w * h < 2**31 and 2 * w * h < 2**32
    T = 3
    fr = _limit_frames(w, h, seed=880 + (w * h) % 16)
    p = O.Params(w, h, tau=0.02)
    o = O.load()
    hist_o = o.histograms_parallel(fr.ctypes.data, T, p)
    so, ko = o.select(hist_o, p)
    dev = torch.from_numpy(fr).cuda()
    del fr
    gc.collect()
    f = NGFF(w, h, tau=0.02, max_frames_per_push=T)
    s, k, hist = f.push(dev, return_hist=True)
    torch.cuda.synchronize()
    f.status()
    hg = hist.cpu().numpy().view(np.uint32)
    assert np.array_equal(hg, hist_o), "histograms at the pixel limit"
    assert (hg.sum(axis=1) == w * h).all() and hg[1, 0] == w * h and hg[2, -1] == w * h
    assert np.array_equal(k.cpu().numpy(), ko)
    sg = s.cpu().numpy().astype(np.float64)
    assert (np.abs(sg - so) <= SCORE_RTOL * so).all(), (sg, so)
    assert sg[2] == 1.0  # L1 = 2N exactly
    f.close()
    del dev
    torch.cuda.empty_cache()


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_spatial_signals_at_the_lowres_limit(kind):
    from paper_2609_03675_gb300 import NGFF
    w = h = 4096  # W·H = 2^24: the low-res L1 numerator 255·W·H just fits 32 bits
    T = 3
    fr = _frames(w, h, T, seed=890 + kind)
    _, so, ko = SO.run(fr, O.Params(w, h, tau=0.01), kind)
    feats = np.stack([SO.features(x, O.Params(w, h), kind) for x in fr])
    f = NGFF(w, h, tau=0.01, signal=kind, max_frames_per_push=T)
    s, k, hist = f.push(torch.from_numpy(fr).cuda(), return_hist=True)
    torch.cuda.synchronize()
    f.status()
    got = hist.cpu().numpy().view(np.uint32)
    if kind == SO.DHASH:
        w64 = got.astype(np.uint64)
        got = np.concatenate([(w64[:, [j]] >> np.arange(32, dtype=np.uint64)) & 1 for j in range(2)], axis=1)
    assert np.array_equal(got.astype(np.int64), feats)
    assert np.array_equal(k.cpu().numpy(), ko)
    sg = s.cpu().numpy().astype(np.float64)
    assert (np.abs(sg - so) <= SCORE_RTOL * so).all()
