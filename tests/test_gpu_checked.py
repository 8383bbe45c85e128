"""The checked build (kernels compiled with -DCOFIE_DEBUG_CHECKS=1, which
check every computed index against their launch arguments and report a
failed check through cofie_ngff_status) run over representative workloads:
the fast and generic histogram kernels (odd sizes, an odd byte offset), the
small-push walk kernel on staged and unstaged rows, one- and two-word gap masks, the
spatial signals on both of their kernels, scene changes across scan tiles,
the frame-order walk (L_max = 0), batches, shards, candidates and gather,
and QER on both scoring kernels.
Every result must still equal the oracle's and no check may fail. A memory
checker is not available on the GPUs this is tested on; these checks stand in
for it. The workloads run in a child process that loads the checked library."""
import os
import subprocess
import sys
import tempfile

import pytest
import torch

pytestmark = pytest.mark.gpu

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import sys
sys.path.insert(0, sys.argv[2])
import numpy as np
import torch
from paper_2609_03675_gb300 import _abi
_abi.LIB_PATH = sys.argv[1]
from paper_2609_03675_gb300 import NGFF
import oracle as O
import synth
from oracle import signals_oracle as SO
from oracle import scd_oracle as SC

assert _abi.load().cofie_ngff_checked_build() == 1, "not the checked library"
RT = 1e-6


def frames(w, h, T, seed, mean=8):
    return synth.generate(synth.medium(seed=seed).with_(width=w, height=h, frames=T, mean_scene_len=mean))


def run(f, fr, chunks):
    dev = torch.from_numpy(fr).cuda()
    ss, ks, off = [], [], 0
    for c in chunks:
        s, k = f.push(dev[off:off + c])
        ss.append(s); ks.append(k); off += c
    torch.cuda.synchronize()
    f.status()  # raises on a failed index check
    return torch.cat(ss).cpu().numpy().astype(np.float64), torch.cat(ks).cpu().numpy()


def same(sg, kg, so, ko, label):
    assert np.array_equal(kg, ko), label
    assert (np.abs(sg - so) <= RT * so).all(), label


n = 0
# histogram: fast kernel (64x48) and generic kernel (37x23); L_max 7/30/40 (one and two mask words); B 32 and 7
for (w, h) in ((64, 48), (37, 23)):
    fr = frames(w, h, 300, seed=600 + w)
    for bins, l_max in ((32, 30), (7, 7), (32, 40)):
        p = O.Params(w, h, bins=bins, tau=0.05, l_max=l_max)
        _, so, ko = O.load().run(fr, p)
        for chunks in ([300], [1, 2, 63, 64, 65, 105]):
            f = NGFF(w, h, bins=bins, tau=0.05, l_max=l_max)
            sg, kg = run(f, fr, chunks)
            same(sg, kg, so, ko, f"hist {w}x{h} B{bins} L{l_max} {chunks[:2]}")
            n += 1
# frames at an odd byte offset (the generic kernel on a pixel count the fast kernel takes), and the
# walk kernel reading 256-bin rows from global memory (too wide to stage) for pushes of 20 frames
fr = frames(64, 48, 120, seed=690)
raw = torch.empty(fr.nbytes + 64, dtype=torch.uint8, device="cuda")
raw[3:3 + fr.nbytes].copy_(torch.from_numpy(fr.reshape(-1)))
_, so, ko = O.load().run(fr, O.Params(64, 48, tau=0.05, l_max=30))
f = NGFF(64, 48, tau=0.05, l_max=30)
s1, k1 = f.push(raw[3:3 + fr.nbytes].view(fr.shape))
torch.cuda.synchronize(); f.status()
same(s1.cpu().numpy().astype(np.float64), k1.cpu().numpy(), so, ko, "generic kernel, offset 3"); n += 1
_, so, ko = O.load().run(fr, O.Params(64, 48, bins=256, tau=0.05, l_max=64))
f = NGFF(64, 48, bins=256, tau=0.05, l_max=64)
same(*run(f, fr, [20] * 6), so, ko, "walk on unstaged 256-bin rows"); n += 1
# spatial signals: streaming cell kernel (64x48) and per-frame kernel (72x40)
for (w, h) in ((64, 48), (72, 40)):
    fr = frames(w, h, 200, seed=640 + w)
    for kind in (SO.LOWRES, SO.DHASH):
        _, so, ko = SO.run(fr, O.Params(w, h, tau=0.05, l_max=11), kind)
        f = NGFF(w, h, tau=0.05, l_max=11, signal=kind)
        sg, kg = run(f, fr, [100, 1, 99])
        same(sg, kg, so, ko, f"signal {kind} {w}x{h}")
        n += 1
# scene changes over several 4096-frame scan tiles; and L_max = 0 (frame-order walk) for two signals
fr = frames(32, 24, 9000, seed=660, mean=40)
hist = np.stack([O.load().histogram(x, O.Params(32, 24)) for x in fr])
so, ko = SC.select(hist, O.Params(32, 24, tau=0.3, l_max=30), 0.05, 0.01)
f = NGFF(32, 24, tau=0.3, l_max=30, signal=_abi.SIGNAL_SCD, scd_cut=0.05, scd_gradual=0.01, max_frames_per_push=9000)
same(*run(f, fr, [9000]), so, ko, "scene changes"); n += 1
_, so, ko = O.load().run(fr, O.Params(32, 24, tau=0.04, l_max=0))
f = NGFF(32, 24, tau=0.04, l_max=0, max_frames_per_push=9000)
same(*run(f, fr, [4000, 1, 4999]), so, ko, "L_max = 0"); n += 1
so, ko = SC.select(hist, O.Params(32, 24, tau=0.3, l_max=0), 0.05, 0.01)
f = NGFF(32, 24, tau=0.3, l_max=0, signal=_abi.SIGNAL_SCD, scd_cut=0.05, scd_gradual=0.01, max_frames_per_push=9000)
same(*run(f, fr, [9000]), so, ko, "scene changes, L_max = 0"); n += 1
# a batch of streams
S = 4
frs = [frames(48, 32, 90, seed=670 + s) for s in range(S)]
f = NGFF(48, 32, tau=0.06, l_max=9, max_streams=S)
dev = [torch.from_numpy(x).cuda() for x in frs]
outs = {s: [] for s in range(S)}
for a, b in ((0, 40), (40, 90)):
    items = []
    for s in range(S):
        sc = torch.empty(b - a, dtype=torch.float32, device="cuda")
        kp = torch.empty(b - a, dtype=torch.uint8, device="cuda")
        items.append((s, dev[s][a:b], sc, kp)); outs[s].append(kp)
    f.push_batch(items)
torch.cuda.synchronize(); f.status()
for s in range(S):
    _, _, ko = O.load().run(frs[s], O.Params(48, 32, tau=0.06, l_max=9))
    assert np.array_equal(torch.cat(outs[s]).cpu().numpy(), ko), f"batch {s}"
n += 1
# shards chained through their gap maps
fr = frames(64, 48, 240, seed=680)
_, so, ko = O.load().run(fr, O.Params(64, 48, tau=0.05, l_max=12))
dev = torch.from_numpy(fr).cuda()
bounds = [0, 50, 51, 170, 240]
maps, hs = {}, {}
for a, b in zip(bounds[:-1], bounds[1:]):
    g = NGFF(64, 48, tau=0.05, l_max=12)
    halo = min(a, 12)
    maps[a] = g.shard_prepare(dev[a - halo:b], n_halo=halo, t0=a).numpy()
    hs[a] = g
gap, ks = 1, []
for a, b in zip(bounds[:-1], bounds[1:]):
    ks.append(hs[a].shard_commit(gap, b - a)[1])
    gap = int(maps[a][gap - 1])
torch.cuda.synchronize()
for g in hs.values():
    g.status()
assert np.array_equal(torch.cat(ks).cpu().numpy(), ko), "shards"
n += 1
# candidates and gather of a closed prefix
f = NGFF(64, 48, tau=0.05, l_max=12)
s, k = f.push(dev)
idx = f.candidates(0)
assert torch.equal(f.candidates_from_keep(k), idx)
out = f.gather(dev, idx)
torch.cuda.synchronize(); f.status()
want = O.load().candidates(ko, 4)
assert np.array_equal(idx.cpu().numpy(), want)
assert torch.equal(out, dev[idx.long()])
n += 1
# QER: the one-SM and the paired kernel, and the benchmark geometry at one wave
from paper_2609_03675_gb300 import QER
from oracle import qer_oracle as Q
from synth import qer as SQ
for spec, kernel in ((SQ.QerSpec(n_text=40, n_heads=8, n_kv_heads=2, head_dim=64, n_frames=6, tokens_per_frame=40,
                                 n_evidence=2, seed=31), 1),
                     (SQ.QerSpec(n_text=64, n_heads=8, n_kv_heads=2, head_dim=64, n_frames=9, tokens_per_frame=24,
                                 n_evidence=2, seed=32), 2),
                     (SQ.QerSpec(n_frames=128), 0)):
    q, k, _ = SQ.generate(spec)
    f = QER(spec.n_text, spec.n_heads, spec.n_kv_heads, spec.head_dim, spec.n_frames, spec.tokens_per_frame, 0.3,
            kernel=kernel)
    w, sel = f.run(torch.from_numpy(q.view(np.int16)).cuda(), torch.from_numpy(k.view(np.int16)).cuda())
    torch.cuda.synchronize()
    f.status()  # raises on a failed layout check
    frames = np.linspace(0, spec.n_frames - 1, min(spec.n_frames, 6)).astype(int)
    w_o = Q.frame_relevance_subset(q, k, spec.tokens_per_frame, frames)
    bound = Q.score_bound(q, k, spec.tokens_per_frame, frames) + 2.0 ** -18 * np.abs(w_o)
    assert np.all(np.abs(w.cpu().numpy()[frames] - w_o) <= bound), f"QER kernel {kernel}"
    n += 1
print("checked workloads", n)
'''


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_checked_build_runs_clean_and_matches_the_oracle():
    sys.path.insert(0, REPO)
    from paper_2609_03675_gb300 import build as B
    d = tempfile.mkdtemp(prefix="cofie_checked_")
    lib = B.build(force=True, defines=["COFIE_DEBUG_CHECKS=1"], out=os.path.join(d, "lib.so"),
                  build_dir=os.path.join(d, "obj"))
    r = subprocess.run([sys.executable, "-c", CHILD, lib, REPO], capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "checked workloads 27" in r.stdout, r.stdout[-2000:]
