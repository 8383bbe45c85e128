"""Failure paths without a GPU fault: an injected device-allocation failure
(host-side hook) and a device wait that runs out (a bounded mbarrier wait
on a phase nothing completes). Each must come back as a status code, leak
nothing, and leave the context and the handle usable."""
import time

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


def _frames(T=40):
    spec = synth.medium(seed=61).with_(width=64, height=48, frames=T, mean_scene_len=7)
    return spec, synth.generate(spec)


def test_injected_allocation_failures_return_enomem_and_leak_nothing():
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    lib = _abi.load()
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    failures = 0
    try:
        for after in range(16):
            lib.cofie_ngff_debug_fail_alloc(after)
            try:
                NGFF(64, 48, signal=_abi.SIGNAL_DHASH).close()  # dHash takes one allocation more
            except NGFFError as e:
                assert e.code == _abi.ENOMEM, e
                failures += 1
            finally:
                lib.cofie_ngff_debug_fail_alloc(-1)
    finally:
        lib.cofie_ngff_debug_fail_alloc(-1)
    assert failures >= 10  # one per allocation of create, then creates succeed
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) <= 4 << 20


def test_staging_allocation_failure_then_recovery():
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    lib = _abi.load()
    spec, fr = _frames()
    host = torch.from_numpy(fr).pin_memory()
    f = NGFF(spec.width, spec.height, tau=0.05)
    lib.cofie_ngff_debug_fail_alloc(0)
    try:
        with pytest.raises(NGFFError) as e:
            f.push(host)
        assert e.value.code == _abi.ENOMEM
    finally:
        lib.cofie_ngff_debug_fail_alloc(-1)
    assert f.frames_seen(0) == 0  # the failed push left the stream unchanged
    s, k = f.push(host)
    torch.cuda.synchronize()
    f.status()
    _, so, ko = O.load().run(fr, O.Params(spec.width, spec.height, tau=0.05))
    assert np.array_equal(k.numpy(), ko)


def test_device_wait_that_runs_out_reports_etimeout():
    from paper_2609_03675_gb300 import NGFF, NGFFError, _abi
    spec, fr = _frames()
    f = NGFF(spec.width, spec.height, tau=0.05)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    f.debug_wait(50_000_000)  # 50 ms
    with pytest.raises(NGFFError) as e:
        f.status()
    waited = time.perf_counter() - t0
    assert e.value.code == _abi.ETIMEOUT
    assert 0.045 <= waited < 5.0, waited
    f.status()  # the error word was read and cleared
    with pytest.raises(NGFFError):
        f.debug_wait(2_000_000_000)  # longer than the 1 s cap: refused on the host
    s, k = f.push(torch.from_numpy(fr).cuda())  # the context and the handle still work
    torch.cuda.synchronize()
    f.status()
    _, so, ko = O.load().run(fr, O.Params(spec.width, spec.height, tau=0.05))
    assert np.array_equal(k.cpu().numpy(), ko)
