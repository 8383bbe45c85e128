"""The C ABI from plain C: tests/c/ngff_client.c (C99, linked against the
library only: no CUDA runtime, no Python) pushes seeded frames from pageable
host memory in uneven pieces and closes the stream after each piece; its
scores and keep codes must equal the oracle's, and each candidate set the
oracle's candidate set of that prefix. The client then pushes the same
frames as two streams through the batched call (pageable host frames and
outputs) and checks both against its single-stream results itself."""
import os
import shutil
import subprocess
import tempfile

import numpy as np
import pytest
import torch

import oracle as O
import synth

pytestmark = pytest.mark.gpu

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def client():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    from paper_2609_03675_gb300 import _abi
    lib_dir = os.path.dirname(_abi.LIB_PATH)
    d = tempfile.mkdtemp(prefix="ngff_client_")
    exe = os.path.join(d, "ngff_client")
    r = subprocess.run(["gcc", "-std=c99", "-O2", "-Wall", "-I", os.path.join(REPO, "include"),
                        os.path.join(REPO, "tests", "c", "ngff_client.c"), "-o", exe, "-L", lib_dir, "-lcofie_ngff",
                        f"-Wl,-rpath,{lib_dir}"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe, d


@pytest.mark.parametrize("tau,l_max", [(0.05, 30), (0.05, 0), (0.3, 7)])
def test_c_client_matches_oracle(client, tau, l_max):
    exe, d = client
    spec = synth.medium(seed=91).with_(width=96, height=64, frames=200, mean_scene_len=10)
    frames = synth.generate(spec)
    fin, fout = os.path.join(d, "in.bin"), os.path.join(d, "out.bin")
    frames.tofile(fin)
    pieces = ["1", "2", "63", "64", "70"]
    r = subprocess.run([exe, fin, fout, str(spec.width), str(spec.height), str(spec.frames), repr(tau), str(l_max),
                        *pieces], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    raw = np.fromfile(fout, dtype=np.uint8)
    T = spec.frames
    scores = raw[: 4 * T].view(np.float32).astype(np.float64)
    keep = raw[4 * T: 5 * T]
    o = O.load()
    _, so, ko = o.run(frames, O.Params(spec.width, spec.height, tau=tau, l_max=l_max))
    assert np.array_equal(keep, ko), np.flatnonzero(keep != ko)[:10]
    assert np.all(np.abs(scores - so) <= 1e-6 * so)
    assert (ko == O.KEEP_NOVELTY).any()
    # the candidate set after each piece: S_c of that prefix (Sec. 3.2 closing safeguards)
    rest = raw[5 * T:].view(np.uint32)
    pos, prefixes = 0, []
    while pos < rest.size:
        t_pre, m = int(rest[pos]), int(rest[pos + 1])
        got_idx = rest[pos + 2: pos + 2 + m]
        want_idx = o.candidates(ko[:t_pre], 4)
        assert np.array_equal(got_idx, want_idx), f"prefix {t_pre}"
        prefixes.append(t_pre)
        pos += 2 + m
    assert prefixes == list(np.cumsum([int(x) for x in pieces]))
