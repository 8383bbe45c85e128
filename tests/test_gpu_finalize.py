"""Closing a prefix on the GPU: the candidate set S_c (last frame, M_min
uniform fill) against the oracle, and the gather of the selected frames
against host-side indexing of the generated frames."""
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


def _ngff(w, h, **kw):
    from paper_2609_03675_gb300 import NGFF
    return NGFF(w, h, **kw)


def test_candidates_small_prefixes_exhaustive():
    o = O.load()
    g = np.random.default_rng(21)
    handles = {m: _ngff(16, 16, m_min=m) for m in range(0, 13)}
    for T in range(1, 41):
        for m_min, f in handles.items():
            for density in (0.0, 0.1, 0.5):
                keep = ((g.random(T) < density) * g.integers(1, 4, size=T)).astype(np.uint8)
                got = f.candidates_from_keep(torch.from_numpy(keep).cuda()).cpu().numpy().astype(np.uint32)
                want = o.candidates(keep, m_min)
                assert np.array_equal(got, want), f"T={T} M_min={m_min} keep={keep}"


@pytest.mark.parametrize("T,density,m_min", [(1023, 0.01, 4), (1024, 0.0, 4), (1025, 0.3, 4), (100_000, 0.05, 4),
                                             (100_000, 0.0, 2000), (65_537, 0.9, 8)])
def test_candidates_long_prefixes(T, density, m_min):
    g = np.random.default_rng(T + m_min)
    keep = ((g.random(T) < density) * g.integers(1, 4, size=T)).astype(np.uint8)
    f = _ngff(16, 16, m_min=m_min)
    got = f.candidates_from_keep(torch.from_numpy(keep).cuda()).cpu().numpy().astype(np.uint32)
    assert np.array_equal(got, O.load().candidates(keep, m_min))


def test_empty_prefix():
    f = _ngff(16, 16)
    assert f.candidates_from_keep(torch.zeros(0, dtype=torch.uint8, device="cuda")).numel() == 0
    assert f.candidates(0).numel() == 0  # a stream with no frames yet


@pytest.mark.parametrize("w,h", [(160, 96), (17, 13)])
def test_push_candidates_gather_pipeline(w, h):
    spec = synth.medium(seed=31).with_(width=w, height=h, frames=120, mean_scene_len=10)
    fr = synth.generate(spec)
    f = _ngff(w, h, tau=0.05, m_min=4)
    dev = torch.from_numpy(fr).cuda()
    f.push(dev)
    idx = f.candidates(0)
    out = f.gather(dev, idx)
    torch.cuda.synchronize()
    f.status()
    _, _, ko = O.load().run(fr, O.Params(w, h, tau=0.05))
    want_idx = O.load().candidates(ko, 4)
    assert np.array_equal(idx.cpu().numpy().astype(np.uint32), want_idx)
    assert np.array_equal(out.cpu().numpy(), fr[want_idx])


def test_gather_rejects_bad_index_without_reading_it():
    from paper_2609_03675_gb300 import NGFFError, _abi
    spec = synth.medium(seed=32).with_(width=64, height=32, frames=10)
    dev = torch.from_numpy(synth.generate(spec)).cuda()
    f = _ngff(64, 32)
    idx = torch.tensor([0, 3, 10, 9], dtype=torch.int32, device="cuda")  # 10 is outside the 10 frames
    out = torch.zeros((4, 32, 64, 3), dtype=torch.uint8, device="cuda")
    f.gather(dev, idx, out=out)
    with pytest.raises(NGFFError) as e:
        f.status()
    assert e.value.code == _abi.EDEVICE
    assert torch.equal(out[[0, 1, 3]], dev[[0, 3, 9]]) and int(out[2].sum()) == 0
    f.status()  # the error word was cleared; the handle keeps working


@pytest.mark.parametrize("w,h", [(160, 96), (17, 13)])
def test_gather_from_pinned_host_frames(w, h):
    """Frames pushed from pinned host memory and gathered from it (the kernel
    reads the host frames through the device's mapping): the same bytes as
    indexing the frames on the host; pageable host frames are refused."""
    from paper_2609_03675_gb300 import NGFFError, _abi
    spec = synth.medium(seed=33).with_(width=w, height=h, frames=150, mean_scene_len=10)
    fr = synth.generate(spec)
    pinned = torch.from_numpy(fr).pin_memory()
    f = _ngff(w, h, tau=0.05, m_min=4)
    f.push(pinned)
    idx = f.candidates(0)
    out = f.gather(pinned, idx)
    torch.cuda.synchronize()
    f.status()
    _, _, ko = O.load().run(fr, O.Params(w, h, tau=0.05))
    want_idx = O.load().candidates(ko, 4)
    assert np.array_equal(idx.cpu().numpy().astype(np.uint32), want_idx)
    assert np.array_equal(out.cpu().numpy(), fr[want_idx])
    # a frame-offset view of the pinned buffer (16-byte aligned only when the frame size is)
    out2 = f.gather(pinned[1:], idx[idx < 149])
    torch.cuda.synchronize()
    f.status()
    assert np.array_equal(out2.cpu().numpy(), fr[1:][want_idx[want_idx < 149]])
    with pytest.raises(NGFFError) as e:
        f.gather(torch.from_numpy(fr), idx)  # pageable host memory
    assert e.value.code == _abi.EINVAL and "pinned host memory" in str(e.value)
