"""cofie_ngff_select_static: selection for callers that may not allocate.

Some callers cannot call cudaMalloc (their device memory belongs to another
framework's pooling allocator under a hard cap, or they are plugins handed
buffers without the right to allocate, or pipelines that fix their memory at
start-up). For them the library offers one entry point whose working tables
live in a static device array. This test calls it through the C ABI twice in
a row, on different streams' histograms, and checks each result against the
regular push entry point (cofie_ngff_push_ex on a fresh stream): keep codes
identical, scores within the same 1e-6 relative tolerance the parity tests
use. It also checks that a size beyond the array is refused with a clear
error. Collected last so that a failure here stops a -x run only after every
other test has run.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _params(lib, _abi, w, h, bins, l_max, tau):
    p = _abi.Params()
    lib.cofie_ngff_default_params(ctypes.byref(p), w, h)
    p.bins, p.l_max, p.tau = bins, l_max, tau
    return p


def test_select_static_matches_push_two_calls_in_a_row():
    from paper_2609_03675_gb300 import NGFF, _abi
    lib = _abi.load()
    cases = [
        (synth.medium(seed=7).with_(width=96, height=64, frames=300), 32, 30, 0.05),
        (synth.medium(seed=8).with_(width=64, height=48, frames=77, mean_scene_len=5), 16, 7, 0.02),
    ]
    stream = torch.cuda.current_stream().cuda_stream
    for spec, bins, l_max, tau in cases:
        frames = torch.from_numpy(synth.generate(spec)).cuda()
        f = NGFF(spec.width, spec.height, bins=bins, l_max=l_max, tau=tau)
        s_ref, k_ref, hist = f.push(frames, return_hist=True)
        n = spec.frames
        s = torch.full((n,), -1.0, dtype=torch.float32, device="cuda")
        k = torch.full((n,), 255, dtype=torch.uint8, device="cuda")
        err = ctypes.create_string_buffer(256)
        p = _params(lib, _abi, spec.width, spec.height, bins, l_max, tau)
        rc = lib.cofie_ngff_select_static(ctypes.byref(p), hist.data_ptr(), n, s.data_ptr(), k.data_ptr(), err,
                                          len(err), stream)
        assert rc == _abi.OK, err.value.decode()
        torch.cuda.synchronize()
        f.status()
        assert torch.equal(k, k_ref), "keep codes differ from cofie_ngff_push_ex"
        sr, sg = s_ref.cpu().numpy().astype(np.float64), s.cpu().numpy().astype(np.float64)
        assert np.all(np.abs(sg - sr) <= 1e-6 * np.abs(sr)), "scores differ from cofie_ngff_push_ex"
        f.close()


def test_select_static_refuses_sizes_beyond_the_array():
    from paper_2609_03675_gb300 import _abi
    lib = _abi.load()
    p = _params(lib, _abi, 64, 48, 32, 30, 0.3)
    err = ctypes.create_string_buffer(256)
    dummy = torch.zeros(1, dtype=torch.int32, device="cuda")
    rc = lib.cofie_ngff_select_static(ctypes.byref(p), dummy.data_ptr(), 33826, None, None, err, len(err), None)
    assert rc == _abi.EINVAL
    assert b"exceeds the static scratch" in err.value
