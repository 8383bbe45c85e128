"""ORACLE for the "scene change detection + H-diff" signal of NGFF's signal
ablation (CoFiE Table "hdiff-signal") -- test infrastructure only.

The paper names the signal and cites the twin-comparison shot-boundary method
of Zhang, Kankanhalli and Smoliar (1993) without defining its thresholds or
how it combines with the histogram difference. The reading restated here:

  H-diff        the histogram rule of Sec. 3.2 unchanged: the C oracle's
                grayscale histograms, the TV distance of Eq. 2, the score
                s = max(s_adj, s_ref) of Eqs. 3-4 and the rule of Eq. 5.
  scene change  twin comparison on the adjacent histogram differences
                SD_t = d(c_t, c_{t-1}) (Eq. 2) with two thresholds T_b
                (cut) and T_s (gradual):
                  SD_t >= T_b            a cut at t; any open run ends (A = 0);
                  T_s <= SD_t < T_b      t joins the run: A_t = A_{t-1} + SD_t;
                  SD_t < T_s             the run ends (A = 0).
                A gradual transition is detected at the frame where the run's
                accumulated difference A first reaches T_b.
  combined      keep(t) = first frame, or novelty (s >= tau_h), or a scene
                change (cut or gradual detection) at t, or the gap rule;
                every kept frame becomes the reference r. Codes: first 3,
                novelty 1, scene change 4, gap 2, drop 0.
  precision     SD and A are integer L1 numerators over 2N; each comparison is
                fp32(numerator) / fp32(2N) >= threshold, as for tau_h.
"""
from __future__ import annotations

import numpy as np

import oracle as O

KEEP_SCENE = 4
HIGH, MID, LOW = 2, 1, 0


def at_least(numerator: int, two_n: int, threshold: float) -> bool:
    """fp32(numerator) / fp32(2N) >= threshold (one IEEE division, round to nearest)."""
    return bool(np.float32(numerator) / np.float32(two_n) >= np.float32(threshold))


def l1(ci: np.ndarray, cj: np.ndarray) -> int:
    """sum_b |c_i[b] - c_j[b]|, the integer numerator of Eq. 2."""
    return int(np.abs(ci.astype(np.int64) - cj.astype(np.int64)).sum())


def classify(a: int, two_n: int, t_cut: float, t_grad: float) -> int:
    if at_least(a, two_n, t_cut):
        return HIGH
    return MID if at_least(a, two_n, t_grad) else LOW


def scene_changes(adj: list[int], two_n: int, t_cut: float, t_grad: float, acc0: int = 0):
    """Twin comparison over adjacent numerators adj[t] (adj[0] unused: frame 0
    has no predecessor and opens no run). Returns (flags, A after the last frame)."""
    flags = np.zeros(len(adj), dtype=bool)
    acc = acc0
    for t in range(1, len(adj)):
        c = classify(adj[t], two_n, t_cut, t_grad)
        if c == HIGH:
            flags[t] = True
            acc = 0
        elif c == MID:
            before = acc
            acc = acc + adj[t]
            flags[t] = at_least(acc, two_n, t_cut) and not at_least(before, two_n, t_cut)
        else:
            acc = 0
    return flags, acc


def select(hist: np.ndarray, p: O.Params, t_cut: float, t_grad: float):
    """(score [T] double, keep codes [T]) of the combined rule."""
    T = hist.shape[0]
    two_n = 2 * p.npix
    score = np.zeros(T)
    keep = np.zeros(T, dtype=np.uint8)
    adj = [0] + [l1(hist[t], hist[t - 1]) for t in range(1, T)]
    scene, _ = scene_changes(adj, two_n, t_cut, t_grad)
    r = 0
    for t in range(T):
        if t == 0:
            keep[0] = O.KEEP_FIRST
            continue
        na, nr = adj[t], l1(hist[t], hist[r])
        score[t] = max(na, nr) / two_n
        if at_least(max(na, nr), two_n, p.tau):
            keep[t] = O.KEEP_NOVELTY
        elif scene[t]:
            keep[t] = KEEP_SCENE
        elif p.l_max > 0 and t - r >= p.l_max:
            keep[t] = O.KEEP_GAP
        if keep[t]:
            r = t
    return score, keep


def run(frames: np.ndarray, p: O.Params, t_cut: float, t_grad: float):
    o = O.load()
    hist = np.stack([o.histogram(f, p) for f in frames]) if len(frames) else np.zeros((0, p.bins), np.uint32)
    score, keep = select(hist, p, t_cut, t_grad)
    return hist, score, keep
