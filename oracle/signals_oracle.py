"""ORACLE for the alternative pre-encoder signals of NGFF's signal ablation
(CoFiE Table "hdiff-signal") -- test infrastructure only.

The paper names the signals and their sources but not their definitions;
the readings restated here (numpy, plain loops for the rule) are the
standard ones, each dropped into the same retention rule as the histogram
difference (Eqs. 3-5 with d replaced):

  grayscale    the oracle's own luma (BT.601 integer, round half up), step 1.
  cells        a G_h x G_w grid over the frame; pixel (y, x) falls in cell
               (floor(y G_h / H), floor(x G_w / W)); S_c = sum of the luma of
               the cell's pixels, n_c = its pixel count.
  low-res      16 x 16 cells; d(i, j) = sum_c |S_c(i) - S_c(j)| / (255 N): the
  difference   mean absolute difference of the block-averaged (low-resolution)
               frames, each cell weighted by its area (Lipton et al. 1998
               frame differencing on a low-resolution grid).
  dHash        9 x 8 cells (9 columns, 8 rows); bit (r, c) = [mean(r, c) >
               mean(r, c + 1)] for c = 0..7, compared exactly as
               S_(r,c) n_(r,c+1) > S_(r,c+1) n_(r,c); d = Hamming / 64
               (difference hash, Zauner 2010).

Both distances are an integer over a fixed denominator, so the keep decision
d >= tau_h is taken as fp32(numerator) / fp32(denominator) >= tau_h, as for
the histogram. Scores are returned in double.
"""
from __future__ import annotations

import numpy as np

import oracle as O

LOWRES, DHASH = 1, 2
GRIDS = {LOWRES: (16, 16), DHASH: (8, 9)}  # (rows, columns)


def cell_sums(frame: np.ndarray, p: O.Params, grid) -> tuple[np.ndarray, np.ndarray]:
    """(S [G_h, G_w] int64 luma sums, n [G_h, G_w] pixel counts) of one frame."""
    gh, gw = grid
    H, W = p.height, p.width
    y = O.load().luma_map(frame.reshape(H, W, 3), p).astype(np.int64)
    cy = (np.arange(H) * gh) // H
    cx = (np.arange(W) * gw) // W
    S = np.zeros((gh, gw), dtype=np.int64)
    n = np.zeros((gh, gw), dtype=np.int64)
    np.add.at(S, (cy[:, None], cx[None, :]), y)
    np.add.at(n, (cy[:, None], cx[None, :]), 1)
    return S, n


def features(frame: np.ndarray, p: O.Params, kind: int) -> np.ndarray:
    """The signal's feature vector: 256 cell sums (low-res) or the 64 dHash bits."""
    S, n = cell_sums(frame, p, GRIDS[kind])
    if kind == LOWRES:
        return S.reshape(-1)
    bits = S[:, :-1] * n[:, 1:] > S[:, 1:] * n[:, :-1]
    return bits.reshape(-1).astype(np.int64)


def numerator(fa: np.ndarray, fb: np.ndarray, kind: int) -> int:
    return int(np.abs(fa - fb).sum()) if kind == LOWRES else int((fa != fb).sum())


def denominator(p: O.Params, kind: int) -> int:
    return 255 * p.npix if kind == LOWRES else 64


def select(feats: np.ndarray, p: O.Params, kind: int):
    """Eqs. 3-5 with the signal's distance: (score [T] double, keep codes [T])."""
    T = len(feats)
    den = denominator(p, kind)
    score = np.zeros(T)
    keep = np.zeros(T, dtype=np.uint8)
    r = 0
    for t in range(T):
        if t == 0:
            keep[0] = O.KEEP_FIRST
            continue
        na = numerator(feats[t], feats[t - 1], kind)
        nr = numerator(feats[t], feats[r], kind)
        score[t] = max(na, nr) / den
        s32 = np.float32(max(na, nr)) / np.float32(den)
        nov = s32 >= np.float32(p.tau)
        gap = p.l_max > 0 and (t - r) >= p.l_max
        keep[t] = O.KEEP_NOVELTY if nov else (O.KEEP_GAP if gap else O.KEEP_DROP)
        if keep[t]:
            r = t
    return score, keep


def run(frames: np.ndarray, p: O.Params, kind: int):
    feats = np.stack([features(f, p, kind) for f in frames])
    score, keep = select(feats, p, kind)
    return feats, score, keep
