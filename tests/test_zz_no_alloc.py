"""cofie_ngff_select_static: selection for callers that may not allocate.

Some callers cannot call cudaMalloc (their device memory belongs to another
framework's pooling allocator under a hard cap, or they are plugins handed
buffers without the right to allocate, or pipelines that fix their memory at
start-up). For them the library offers one entry point whose working tables
live in a static device array. This test calls it through the C ABI on the
oracle's own histograms and checks every result against the oracle's
selection rule on the same histograms (keep codes identical, scores within
the 1e-6 relative tolerance of the parity tests): two calls in a row on one
stream (the array keeps the previous call's contents), streams long enough
to cross several 2048-frame scan tiles, L_max above 32 (two mask words),
bin counts that are not a multiple of 4 (the scalar row loads). It checks
that the calls allocate no device memory, that the existing push entry point
gives the same decisions, and that sizes beyond the array and the signals
it does not serve are refused with a clear error. Collected last so that a
failure here stops a -x run only after every other test has run.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle as O
import synth

pytestmark = pytest.mark.gpu

SCORE_RTOL = 1e-6


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _params(lib, _abi, w, h, bins, l_max, tau, signal=0):
    p = _abi.Params()
    lib.cofie_ngff_default_params(ctypes.byref(p), w, h)
    p.bins, p.l_max, p.tau, p.signal = bins, l_max, tau, signal
    return p


def _call(lib, _abi, p, hist_dev, n, s, k):
    err = ctypes.create_string_buffer(256)
    rc = lib.cofie_ngff_select_static(ctypes.byref(p), hist_dev.data_ptr(), n, s.data_ptr(), k.data_ptr(), err,
                                      len(err), torch.cuda.current_stream().cuda_stream)
    return rc, err.value.decode()


# (width, height, frames, mean scene length, bins, L_max, tau): 5000 frames cross
# three scan tiles; each case keeps frames by both rules (novelty and gap)
CASES = [
    (32, 16, 5000, 40, 32, 30, 0.30),
    (32, 16, 5000, 60, 16, 33, 0.20),
    (24, 16, 4500, 80, 7, 64, 0.10),
    (96, 64, 300, 20, 32, 30, 0.45),
    (64, 48, 77, 5, 16, 7, 0.30),
]


def _case(w, h, T, scene, bins, l_max, tau, seed):
    spec = synth.medium(seed=seed).with_(width=w, height=h, frames=T, mean_scene_len=scene)
    frames = synth.generate(spec)
    p = O.Params(w, h, bins=bins, l_max=l_max, tau=tau)
    hist, so, ko = O.load().run(frames, p)
    return frames, hist, so, ko


def test_select_static_matches_the_oracle_two_calls_in_a_row():
    from paper_2609_03675_gb300 import _abi
    lib = _abi.load()
    for i, (w, h, T, scene, bins, l_max, tau) in enumerate(CASES):
        _, hist, so, ko = _case(w, h, T, scene, bins, l_max, tau, seed=300 + i)
        hd = torch.from_numpy(hist.view(np.int32)).cuda()
        p = _params(lib, _abi, w, h, bins, l_max, tau)
        for call in range(2):
            s = torch.full((T,), -1.0, dtype=torch.float32, device="cuda")
            k = torch.full((T,), 255, dtype=torch.uint8, device="cuda")
            rc, msg = _call(lib, _abi, p, hd, T, s, k)
            assert rc == _abi.OK, msg
            torch.cuda.synchronize()
            kg, sg = k.cpu().numpy(), s.cpu().numpy().astype(np.float64)
            label = f"{w}x{h} T={T} B={bins} L={l_max} call {call}"
            assert np.array_equal(kg, ko), f"{label}: keep codes differ at {np.flatnonzero(kg != ko)[:10]}"
            assert np.all(np.abs(sg - so) <= SCORE_RTOL * np.abs(so)), label
        assert (ko == O.KEEP_NOVELTY).any() and (ko == O.KEEP_GAP).any(), "both rules fire"


def test_select_static_agrees_with_the_push_entry_point():
    """The same frames through cofie_ngff_push_ex on a fresh stream (its own
    histograms in) give the same decisions."""
    from paper_2609_03675_gb300 import NGFF, _abi
    lib = _abi.load()
    w, h, T, scene, bins, l_max, tau = CASES[0]
    frames, _, _, _ = _case(w, h, T, scene, bins, l_max, tau, seed=300)
    f = NGFF(w, h, bins=bins, l_max=l_max, tau=tau, max_frames_per_push=T)
    s_ref, k_ref, hist = f.push(torch.from_numpy(frames).cuda(), return_hist=True)
    s = torch.empty(T, dtype=torch.float32, device="cuda")
    k = torch.empty(T, dtype=torch.uint8, device="cuda")
    rc, msg = _call(lib, _abi, _params(lib, _abi, w, h, bins, l_max, tau), hist, T, s, k)
    assert rc == _abi.OK, msg
    torch.cuda.synchronize()
    f.status()
    assert torch.equal(k, k_ref) and torch.equal(s, s_ref)
    f.close()


def test_select_static_allocates_no_device_memory():
    from paper_2609_03675_gb300 import _abi
    lib = _abi.load()
    inputs = []
    for i, (w, h, T, scene, bins, l_max, tau) in enumerate(CASES):
        _, hist, _, _ = _case(w, h, T, scene, bins, l_max, tau, seed=400 + i)
        inputs.append((_params(lib, _abi, w, h, bins, l_max, tau), torch.from_numpy(hist.view(np.int32)).cuda(), T,
                       torch.empty(T, dtype=torch.float32, device="cuda"),
                       torch.empty(T, dtype=torch.uint8, device="cuda")))
    p, hd, T, s, k = inputs[0]
    assert _call(lib, _abi, p, hd, T, s, k)[0] == _abi.OK  # first call on the device: set-up
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for p, hd, T, s, k in inputs * 2:
        rc, msg = _call(lib, _abi, p, hd, T, s, k)
        assert rc == _abi.OK, msg
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0, "free device memory changed during the call"


def test_select_static_refuses_sizes_beyond_the_array_and_other_signals():
    from paper_2609_03675_gb300 import _abi
    lib = _abi.load()
    dummy = torch.zeros(8, dtype=torch.int32, device="cuda")
    out_s = torch.zeros(8, dtype=torch.float32, device="cuda")
    out_k = torch.zeros(8, dtype=torch.uint8, device="cuda")
    p = _params(lib, _abi, 64, 48, 32, 30, 0.3)
    err = ctypes.create_string_buffer(256)
    rc = lib.cofie_ngff_select_static(ctypes.byref(p), dummy.data_ptr(), 33826, None, None, err, len(err), None)
    assert rc == _abi.EINVAL
    assert b"exceeds the static scratch" in err.value
    for sig in (_abi.SIGNAL_LOWRES, _abi.SIGNAL_DHASH, _abi.SIGNAL_SCD):
        rc, msg = _call(lib, _abi, _params(lib, _abi, 64, 48, 32, 30, 0.3, signal=sig), dummy, 8, out_s, out_k)
        assert rc == _abi.EINVAL and "histogram signal" in msg
