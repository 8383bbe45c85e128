"""The C-ABI library builds, loads without a GPU, exports every declared
symbol, and rejects bad parameters before touching the device."""
import ctypes
import os
import re

import pytest

from tests.conftest import REPO

HEADER = os.path.join(REPO, "include", "cofie_ngff.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cofie_(?:ngff|qer)_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_03675_gb300 import build
    build.build()
    from paper_2609_03675_gb300 import _abi
    return _abi.load()


def test_exports_every_declared_symbol(lib):
    from paper_2609_03675_gb300 import _abi
    names = _declared()
    assert len(names) >= 10
    assert sorted(_abi.EXPORTS) == names, "binding and header disagree"
    for n in names:
        assert hasattr(lib, n), f"{n} not exported"


def test_param_struct_layout_matches_header(lib):
    from paper_2609_03675_gb300 import _abi
    # width..luma_den: 10 x 4 bytes, max_streams, max_frames_per_push, device, pad, u64, signal, scd_cut,
    # scd_gradual, max_stream_frames
    assert ctypes.sizeof(_abi.Params) == 80
    assert ctypes.sizeof(_abi.PushDesc) == 32


def test_defaults_are_the_papers(lib):
    import json
    from paper_2609_03675_gb300 import _abi
    p = _abi.Params()
    lib.cofie_ngff_default_params(ctypes.byref(p), 1920, 1080)
    d = json.load(open(os.path.join(REPO, "tests", "golden", "ngff_defaults.json")))
    assert (p.bins, p.m_min, p.l_max) == (d["bins"]["value"], d["m_min"]["value"], d["l_max"]["value"])
    assert abs(p.tau - d["tau_h"]["value"]) < 1e-7
    assert list(p.luma_w) == [299, 587, 114] and p.luma_den == 1000
    assert p.max_stream_frames == 1 << 20  # the retention record's default reach (not from the paper)


@pytest.mark.parametrize("field,value,msg", [
    ("width", 0, "width"), ("bins", 0, "bins"), ("bins", 257, "bins"),
    ("l_max", 257, "l_max"), ("tau", float("nan"), "NaN"), ("luma_den", 999, "sum"), ("max_streams", 0, "streams"),
    ("max_frames_per_push", 0, "max_frames"),
])
def test_create_rejects_bad_params_without_gpu(lib, field, value, msg):
    from paper_2609_03675_gb300 import _abi
    p = _abi.Params()
    lib.cofie_ngff_default_params(ctypes.byref(p), 64, 48)
    setattr(p, field, value)
    h = ctypes.c_void_p()
    rc = lib.cofie_ngff_create(ctypes.byref(p), ctypes.byref(h))
    assert rc == _abi.EINVAL
    assert msg in lib.cofie_ngff_global_error().decode()
    assert not h.value


def test_null_handle_calls_are_rejected(lib):
    from paper_2609_03675_gb300 import _abi
    assert lib.cofie_ngff_push(None, 0, None, 0, None, None, None) == _abi.EINVAL
    assert lib.cofie_ngff_reset(None, 0, None) == _abi.EINVAL
    assert lib.cofie_ngff_status(None, None) == _abi.EINVAL
    m = ctypes.c_uint32(7)
    assert lib.cofie_ngff_candidates(None, 0, None, 0, ctypes.addressof(m), None) == _abi.EINVAL
    assert lib.cofie_ngff_candidates_from_keep(None, None, 0, None, ctypes.addressof(m), None) == _abi.EINVAL
    assert m.value == 7
    assert lib.cofie_ngff_last_error(None) == b""
    lib.cofie_ngff_destroy(None)


@pytest.mark.parametrize("width,height,signal,msg", [
    (64, 48, 4, "signal"), (15, 48, 1, "low-res"), (64, 15, 1, "low-res"), (4097, 4097, 1, "low-res"),
    (8, 48, 2, "dHash"), (64, 7, 2, "dHash"), (46341, 46340, 2, "too large"),
])
def test_create_rejects_bad_signal_shapes(lib, width, height, signal, msg):
    from paper_2609_03675_gb300 import _abi
    p = _abi.Params()
    lib.cofie_ngff_default_params(ctypes.byref(p), width, height)
    p.signal = signal
    h = ctypes.c_void_p()
    assert lib.cofie_ngff_create(ctypes.byref(p), ctypes.byref(h)) == _abi.EINVAL
    assert msg in lib.cofie_ngff_global_error().decode()
    assert not h.value


@pytest.mark.parametrize("field", ["scd_cut", "scd_gradual"])
def test_create_rejects_nan_scene_thresholds(lib, field):
    from paper_2609_03675_gb300 import _abi
    p = _abi.Params()
    lib.cofie_ngff_default_params(ctypes.byref(p), 64, 48)
    assert (p.scd_cut, p.scd_gradual) == (pytest.approx(0.30), pytest.approx(0.10))
    p.signal = _abi.SIGNAL_SCD
    setattr(p, field, float("nan"))
    h = ctypes.c_void_p()
    assert lib.cofie_ngff_create(ctypes.byref(p), ctypes.byref(h)) == _abi.EINVAL
    assert "NaN" in lib.cofie_ngff_global_error().decode()


@pytest.mark.parametrize("field,value,msg", [
    ("n_text", 0, "n_text"), ("n_text", 4097, "n_text"), ("n_kv_heads", 3, "divide"), ("head_dim", 36, "multiple of 64"),
    ("rho", 1.5, "rho"), ("kernel", 3, "kernel"), ("max_frames", 0, "max_frames"),
])
def test_qer_create_rejects_bad_params_without_gpu(lib, field, value, msg):
    """QER's parameters are validated before any CUDA call: n_text runs to
    4096 (scored in passes of at most 256), n_kv_heads divides n_heads,
    H_kv * d_h is a multiple of 64, rho lies in [0, 1]."""
    from paper_2609_03675_gb300 import _abi
    p = _abi.QerParams(256, 32, 8, 128, 16, 256, 0.3, -1, 0)
    setattr(p, field, value)
    h = ctypes.c_void_p()
    assert lib.cofie_qer_create(ctypes.byref(p), ctypes.byref(h)) == _abi.EINVAL
    assert msg in lib.cofie_qer_last_error(None).decode()
    assert not h.value


def test_header_is_c99_and_a_c_client_links(tmp_path):
    """include/cofie_ngff.h compiles as C99 (warnings are errors) and a C
    client links against the library alone."""
    import shutil
    import subprocess
    from paper_2609_03675_gb300 import _abi
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    lib_dir = os.path.dirname(_abi.LIB_PATH)
    exe = tmp_path / "ngff_client"
    r = subprocess.run(["gcc", "-std=c99", "-O2", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(REPO, "include"),
                        os.path.join(REPO, "tests", "c", "ngff_client.c"), "-o", str(exe), "-L", lib_dir,
                        "-lcofie_ngff", f"-Wl,-rpath,{lib_dir}"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """No fallback: with the library absent, creating a handle raises an error
    that says how to build it (nothing runs on the CPU instead)."""
    from paper_2609_03675_gb300 import NGFF, QER, _abi
    monkeypatch.setattr(_abi, "LIB_PATH", str(tmp_path / "libcofie_ngff.so"))
    monkeypatch.setattr(_abi, "_lib", None)
    with pytest.raises(RuntimeError, match="has not been built"):
        NGFF(64, 48)
    with pytest.raises(RuntimeError, match="has not been built"):
        QER(8, 32, 8, 128, 4, 16, 0.3)
