"""Helpers for the GPU parity tests: run the library through its C ABI and
compare with the oracle on the same seeded frames."""
from __future__ import annotations

import numpy as np
import torch

import oracle as O

SCORE_RTOL = 1e-6  # fp32 score against the oracle's double-precision distance


def run_stream(f, frames_dev: torch.Tensor, chunks, stream: int = 0):
    """Pushes frames_dev in pieces of the given sizes; returns numpy (hist, scores, keep)."""
    hs, ss, ks = [], [], []
    off = 0
    for c in chunks:
        s, k, h = f.push(frames_dev[off:off + c], stream, return_hist=True)
        hs.append(h)
        ss.append(s)
        ks.append(k)
        off += c
    assert off == frames_dev.shape[0]
    torch.cuda.synchronize()
    f.status()
    cat = (lambda xs, d: torch.cat(xs).cpu().numpy() if xs else np.zeros((0,), d))
    return (cat(hs, np.int32).view(np.uint32).reshape(-1, f.feature_words), cat(ss, np.float32),
            cat(ks, np.uint8))


def assert_parity(got, want, tau: float, label: str = ""):
    """Histograms bit-exact, scores within SCORE_RTOL, keep codes identical.

    Returns the frames whose oracle score lies within SCORE_RTOL of tau (the
    tolerance band). The keep decision is taken in fp32 on both sides, so the
    masks must agree on those frames too."""
    hg, sg, kg = got
    ho, so, ko = want
    assert hg.shape == ho.shape, label
    bad = np.flatnonzero((hg != ho).any(axis=1)) if hg.size else []
    assert len(bad) == 0, f"{label}: histograms differ at frames {list(bad[:10])}"
    err = np.abs(sg.astype(np.float64) - so)
    lim = SCORE_RTOL * np.abs(so)
    badscore = np.flatnonzero(err > lim)
    assert len(badscore) == 0, f"{label}: scores differ at {list(badscore[:10])}: {sg[badscore[:5]]} vs {so[badscore[:5]]}"
    band = np.flatnonzero(np.abs(so - tau) <= SCORE_RTOL * max(abs(tau), 1e-30))
    badkeep = np.flatnonzero(kg != ko)
    assert len(badkeep) == 0, f"{label}: keep codes differ at {list(badkeep[:10])} (band frames {list(band)})"
    return band


def oracle_run(frames_np: np.ndarray, p: O.Params):
    return O.load().run(frames_np, p)
