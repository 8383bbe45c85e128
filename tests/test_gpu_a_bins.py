"""Device binning of every RGB triple, checked before any histogram kernel runs.

The fast histogram kernel's per-pixel grayscale (two dp2a per pixel) and bin
(one multiply-high) functions are applied by a diagnostic kernel that only
writes one byte per pixel, so a wrong bin shows up here as a mismatch rather
than as a counter index outside the kernel's shared-memory table. This file
is collected first among the GPU tests.
"""
import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu


def _ngff(w, h, **kw):
    from paper_2609_03675_gb300 import NGFF
    return NGFF(w, h, **kw)


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_every_rgb_triple_bins_on_device():
    """The fast kernel's per-pixel grayscale + bin functions on all 2^24 triples."""
    v = torch.arange(1 << 24, dtype=torch.int64)
    px = torch.stack([(v >> 16) & 255, (v >> 8) & 255, v & 255], -1).to(torch.uint8)
    y = torch.from_numpy(O.load().luma_map(px.numpy(), O.Params(8, 8)).astype(np.int64))
    dev = px.cuda()
    for bins in (32, 256, 24, 7):
        f = _ngff(16, 16, bins=bins)
        got = f.debug_bins(dev).cpu().to(torch.int64)
        want = torch.from_numpy(np.array([O.load().bin_of(i, bins) for i in range(256)], dtype=np.int64))[y]
        assert torch.equal(got, want), f"bins={bins}"
