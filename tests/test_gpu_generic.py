"""The generic histogram kernel: frames whose pixel count is not a multiple
of 16, or that start at any byte offset (the bulk-copy kernel needs both),
against the oracle: histograms bit-exact, scores within 1e-6 relative, keep
codes identical. Covers every frame alignment mod 16, the three bin paths
(one multiply-high, two-step, plain division when no multiply-high verifies)
and a frame of many CTA slices (1917 x 1080) with its ragged edges."""
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


def _at_offset(fr: np.ndarray, off: int) -> torch.Tensor:
    """The frames copied to a device buffer starting `off` bytes past a 256-byte boundary."""
    raw = torch.empty(fr.nbytes + 256, dtype=torch.uint8, device="cuda")
    raw[off:off + fr.nbytes].copy_(torch.from_numpy(fr.reshape(-1)))
    return raw[off:off + fr.nbytes].view(fr.shape)


@pytest.mark.parametrize("w,h", [(17, 13), (64, 48), (33, 1), (5, 3), (1, 1)])
def test_every_frame_alignment(w, h):
    from paper_2609_03675_gb300 import NGFF
    spec = synth.medium(seed=w * 31 + h).with_(width=w, height=h, frames=40, mean_scene_len=5)
    fr = synth.generate(spec)
    p = O.Params(w, h, tau=0.05)
    want = oracle_run(fr, p)
    for off in range(16):
        f = NGFF(w, h, tau=0.05)
        got = run_stream(f, _at_offset(fr, off), [1, 7, 32])
        assert_parity(got, want, 0.05, f"{w}x{h} offset {off}")
        f.close()


@pytest.mark.parametrize("bins,luma_w,luma_den", [(32, (299, 587, 114), 1000), (7, (299, 587, 114), 1000),
                                                  (7, (1, 0, 0), 1), (256, (77, 150, 29), 256)])
def test_bin_paths(bins, luma_w, luma_den):
    from paper_2609_03675_gb300 import NGFF
    w, h = 45, 29
    spec = synth.medium(seed=bins + luma_den).with_(width=w, height=h, frames=60, mean_scene_len=6)
    fr = synth.generate(spec)
    p = O.Params(w, h, bins=bins, tau=0.05, luma_w=luma_w, luma_den=luma_den)
    want = oracle_run(fr, p)
    f = NGFF(w, h, bins=bins, tau=0.05, luma_weights=luma_w, luma_den=luma_den)
    got = run_stream(f, _at_offset(fr, 5), [60])
    assert_parity(got, want, 0.05, f"B={bins} luma {luma_w}/{luma_den}")
    f.close()


def test_many_slices_per_frame():
    """1917 x 1080 (2,070,360 pixels: 64 CTA slices per frame and a ragged
    epilogue), at an offset that leaves a prologue too."""
    from paper_2609_03675_gb300 import NGFF
    spec = synth.hd1080().with_(width=1917, height=1080, frames=24)
    fr = synth.generate(spec)
    o = O.load()
    p = O.Params(spec.width, spec.height)
    hist_o = o.histograms_parallel(fr.ctypes.data, spec.frames, p)
    so, ko = o.select(hist_o, p)
    for off in (0, 3, 10):
        f = NGFF(spec.width, spec.height)
        got = run_stream(f, _at_offset(fr, off), [24])
        assert_parity(got, (hist_o, so, ko), 0.30, f"1917x1080 offset {off}")
        f.close()
