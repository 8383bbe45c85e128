"""Pins that tie the NGFF oracle to facts other than itself.

Each ``pin_*`` takes a loaded ``oracle.Oracle`` and raises AssertionError when
the oracle disagrees with what the paper or the mathematics fixes:

* luma: every one of the 2^24 RGB triples against ITU-R BT.601's decimal
  weights evaluated in numpy double precision, plus the textbook luma of the
  100% colour-bar primaries and secondaries (tests/golden/bt601_colour_bars.txt);
* binning: numpy.histogram's binning of Y/255 over [0, 1] (B dividing 256)
  and of Y over [0, 256) (any B);
* histograms: numpy.histogram of independently computed intensities, the
  pixel-count sum, one-hot constant frames, pixel-permutation invariance;
* Eq. 2: closed forms (0 on identical, 1 on disjoint supports, exact dyadic
  values), symmetry, triangle inequality, the changed-pixel bound,
  invariance to translation with wrap-around;
* Eqs. 3-5: special cases that reduce to closed forms (tau <= 0 keeps all,
  tau > 1 keeps exactly 0, L_max, 2 L_max, ...), constructed streams where
  only the adjacent term or only the reference term crosses tau, an exact
  tie at tau (">="), causality (prefix runs agree), seeded hard cuts kept,
  and brute force over all 2^4 keep masks of random 4-frame 8x8 streams;
* the closing safeguards: set properties and numpy's linspace for the
  uniformly spaced fill.

``main(path)`` runs every pin against the oracle library at ``path`` and
returns the number of failing pins (used to check that mutated oracles are
caught).
"""
from __future__ import annotations

import json
import os
import sys
import traceback

import numpy as np

_REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if _REPO not in sys.path:
    sys.path.insert(0, _REPO)

import oracle as O  # noqa: E402
import synth  # noqa: E402

GOLDEN = os.path.join(_REPO, "tests", "golden")


# --------------------------------------------------------------- helpers --

def np_luma(px: np.ndarray) -> np.ndarray:
    """BT.601 luma 0.299 R + 0.587 G + 0.114 B, rounded half up, evaluated in
    double. The exact value has three decimals, so a 1e-6 nudge resolves the
    .5 ties upward without touching any other value."""
    f = px.astype(np.float64)
    x = 0.299 * f[..., 0] + 0.587 * f[..., 1] + 0.114 * f[..., 2]
    return np.floor(x + 0.5 + 1e-6).astype(np.int64)


def np_hist(frame: np.ndarray, bins: int) -> np.ndarray:
    y = np_luma(frame.reshape(-1, 3))
    return np.histogram(y, bins=bins, range=(0, 256))[0].astype(np.int64)


def _rng(seed):
    return np.random.default_rng(seed)


# ------------------------------------------------------------------ luma --

def pin_luma_exhaustive(o):
    p = O.Params(8, 8)
    v = np.arange(1 << 24, dtype=np.uint32)
    ties = 0
    for lo in range(0, 1 << 24, 1 << 21):
        c = v[lo:lo + (1 << 21)]
        px = np.stack([(c >> 16) & 255, (c >> 8) & 255, c & 255], -1).astype(np.uint8)
        y = o.luma_map(px, p).astype(np.int64)
        f = px.astype(np.float64)
        x = 0.299 * f[:, 0] + 0.587 * f[:, 1] + 0.114 * f[:, 2]
        frac = x - np.floor(x)
        tie = np.abs(frac - 0.5) < 1e-9
        ties += int(tie.sum())
        assert np.array_equal(y[~tie], np.floor(x[~tie] + 0.5).astype(np.int64)), "luma off a tie"
        # at an exact .5 the rounding goes up
        assert np.array_equal(y[tie], np.floor(x[tie]).astype(np.int64) + 1), "luma at a tie"
    assert ties > 0, "no rounding ties exercised"


def pin_luma_colour_bars(o):
    p = O.Params(8, 8)
    with open(os.path.join(GOLDEN, "bt601_colour_bars.txt")) as fh:
        rows = [ln.split() for ln in fh if ln.strip() and not ln.startswith("#")]
    assert len(rows) >= 8
    for name, r, g, b, y in rows:
        assert o.luma(int(r), int(g), int(b), p) == int(y), f"luma of {name}"
    for v in range(256):
        assert o.luma(v, v, v, p) == v, "gray must map to itself"


# ---------------------------------------------------------------- binning --

def pin_bins_numpy(o):
    ys = np.arange(256)
    for B in (1, 2, 4, 8, 16, 32, 64, 128, 256):
        for y in ys:
            h = np.histogram([y / 255.0], bins=B, range=(0.0, 1.0))[0]
            assert o.bin_of(int(y), B) == int(np.argmax(h)), f"bin of {y} among {B} (unit range)"
    for B in (3, 7, 24, 48, 100, 255):
        for y in ys:
            h = np.histogram([y], bins=B, range=(0, 256))[0]
            assert o.bin_of(int(y), B) == int(np.argmax(h)), f"bin of {y} among {B} ([0,256) range)"


# ------------------------------------------------------------- histogram --

def pin_histogram_numpy(o):
    g = _rng(11)
    for (w, h) in ((1, 1), (7, 5), (33, 17), (64, 48)):
        for B in (1, 3, 32, 100, 256):
            f = g.integers(0, 256, size=(h, w, 3), dtype=np.uint8)
            got = o.histogram(f, O.Params(w, h, bins=B)).astype(np.int64)
            assert np.array_equal(got, np_hist(f, B)), f"histogram {w}x{h} B={B}"


def pin_histogram_invariants(o):
    g = _rng(12)
    w, h = 40, 30
    p = O.Params(w, h)
    for _ in range(20):
        f = g.integers(0, 256, size=(h, w, 3), dtype=np.uint8)
        c = o.histogram(f, p)
        assert int(c.sum()) == w * h, "histogram must sum to W*H"
        perm = g.permutation(w * h)
        fp = f.reshape(-1, 3)[perm].reshape(h, w, 3)
        assert np.array_equal(o.histogram(fp, p), c), "pixel permutation changed the histogram"
    for _ in range(20):
        col = g.integers(0, 256, size=3)
        f = np.empty((h, w, 3), dtype=np.uint8)
        f[...] = col
        c = o.histogram(f, p)
        k = int(np_luma(col.reshape(1, 3))[0]) * 32 // 256
        expect = np.zeros(32, dtype=np.uint32)
        expect[k] = w * h
        assert np.array_equal(c, expect), "constant frame must be one-hot"


# ------------------------------------------------------------------ Eq. 2 --

def pin_tv_closed_forms(o):
    N = 1000
    a = np.array([N, 0, 0, 0], dtype=np.uint32)
    b = np.array([0, N, 0, 0], dtype=np.uint32)
    assert o.tv(a, a, N) == 0.0
    assert o.tv(a, b, N) == 1.0, "disjoint supports are at distance 1"
    c = np.array([N // 2, N // 2, 0, 0], dtype=np.uint32)
    d = np.array([N // 2, 0, N // 2, 0], dtype=np.uint32)
    assert o.tv(c, d, N) == 0.5 and o.tv32(c, d, N) == 0.5
    e = np.array([N // 4, N // 4, N // 4, N // 4], dtype=np.uint32)
    assert o.tv(a, e, N) == 0.75 and o.tv32(a, e, N) == 0.75
    g = _rng(13)
    for _ in range(200):
        B = int(g.integers(1, 40))
        hs = [np.bincount(g.integers(0, B, size=N), minlength=B).astype(np.uint32) for _ in range(3)]
        x, y, z = (o.tv(hs[0], hs[1], N), o.tv(hs[1], hs[2], N), o.tv(hs[0], hs[2], N))
        assert 0.0 <= x <= 1.0
        assert x == o.tv(hs[1], hs[0], N), "symmetry"
        assert z <= x + y + 1e-12, "triangle inequality"
        t32 = o.tv32(hs[0], hs[1], N)
        assert abs(t32 - x) <= 2.0 ** -23 * max(x, 1e-30) + 1e-15, "fp32 decision value off the distance"


def pin_tv_frame_bounds(o):
    g = _rng(14)
    w, h = 48, 32
    N = w * h
    p = O.Params(w, h)
    for _ in range(20):
        f = g.integers(0, 256, size=(h, w, 3), dtype=np.uint8)
        k = int(g.integers(1, N))
        f2 = f.copy().reshape(-1, 3)
        idx = g.choice(N, size=k, replace=False)
        f2[idx] = g.integers(0, 256, size=(k, 3), dtype=np.uint8)
        f2 = f2.reshape(h, w, 3)
        d = o.tv(o.histogram(f, p), o.histogram(f2, p), N)
        assert d <= k / N + 1e-12, "distance exceeds the changed-pixel fraction"
        sh = np.roll(f, shift=(int(g.integers(0, h)), int(g.integers(0, w))), axis=(0, 1))
        assert o.tv(o.histogram(f, p), o.histogram(sh, p), N) == 0.0, "translation with wrap is a permutation"


# -------------------------------------------------------------- Eqs. 3-5 --

def _hist_stream(rows):
    return np.array(rows, dtype=np.uint32)


def pin_rule_thresholds(o):
    g = _rng(15)
    for _ in range(10):
        T = int(g.integers(2, 70))
        B = 8
        hist = np.stack([np.bincount(g.integers(0, B, size=100), minlength=B) for _ in range(T)]).astype(np.uint32)
        for L in (1, 2, 3, 7, 30):
            p = O.Params(10, 10, bins=B, l_max=L, tau=0.0)
            score, keep = o.select(hist, p)
            assert keep[0] == O.KEEP_FIRST and score[0] == 0.0
            assert (keep[1:] == O.KEEP_NOVELTY).all(), "tau = 0 keeps every frame by novelty"
            p = O.Params(10, 10, bins=B, l_max=L, tau=1.5)
            score, keep = o.select(hist, p)
            kept = np.flatnonzero(keep)
            assert np.array_equal(kept, np.arange(0, T, L)), "tau > 1 keeps exactly 0, L, 2L, ..."
            assert (keep[kept[1:]] == O.KEEP_GAP).all()
            assert ((score >= 0) & (score <= 1)).all()
        # L_max = 0 turns the forced retention off: with tau > 1 only the first frame is kept
        _, keep = o.select(hist, O.Params(10, 10, bins=B, l_max=0, tau=1.5))
        assert np.array_equal(np.flatnonzero(keep), [0])
        _, keep = o.select(hist, O.Params(10, 10, bins=B, l_max=0, tau=0.0))
        assert (keep[1:] == O.KEEP_NOVELTY).all()
    # a constant stream scores zero everywhere
    hist = np.tile(np.array([[100, 0, 0, 0]], dtype=np.uint32), (40, 1))
    score, keep = o.select(hist, O.Params(10, 10, bins=4, l_max=7, tau=0.1))
    assert (score == 0).all() and np.array_equal(np.flatnonzero(keep), np.arange(0, 40, 7))
    _, keep = o.select(hist, O.Params(10, 10, bins=4, l_max=0, tau=0.1))
    assert np.array_equal(np.flatnonzero(keep), [0]), "no forced retention: a constant stream keeps its first frame"


def pin_rule_terms(o):
    # only the reference term crosses tau: slow drift of 0.1 per frame
    hist = _hist_stream([[100 - 10 * t, 10 * t] for t in range(8)])
    score, keep = o.select(hist, O.Params(10, 10, bins=2, l_max=100, tau=0.25))
    assert np.array_equal(np.flatnonzero(keep), [0, 3, 6]), "accumulated drift must trigger via s_ref"
    assert np.allclose(score[1:], [0.1, 0.2, 0.3, 0.1, 0.2, 0.3, 0.1])
    # only the adjacent term crosses tau: X and Y are both 0.25 from the reference
    A, X, Y = [50, 25, 25], [50, 50, 0], [50, 0, 50]
    score, keep = o.select(_hist_stream([A, X, Y]), O.Params(10, 10, bins=3, l_max=100, tau=0.4))
    assert list(keep) == [O.KEEP_FIRST, O.KEEP_DROP, O.KEEP_NOVELTY], "abrupt change must trigger via s_adj"
    assert score[1] == 0.25 and score[2] == 0.5
    # ">=": a distance exactly equal to tau is retained, the next float above is not
    hist = _hist_stream([[50, 50, 0], [50, 0, 50]])
    _, keep = o.select(hist, O.Params(10, 10, bins=3, l_max=100, tau=0.5))
    assert keep[1] == O.KEEP_NOVELTY, "s == tau must be retained"
    _, keep = o.select(hist, O.Params(10, 10, bins=3, l_max=100, tau=float(np.nextafter(np.float32(0.5), np.float32(1)))))
    assert keep[1] == O.KEEP_DROP
    # a gap-retained frame becomes the reference: with L_max = 2 frame 2 is
    # kept by the gap rule, so frame 3 is compared with it (distance 0.2 < tau)
    hist = _hist_stream([[100, 0], [100, 0], [80, 20], [60, 40]])
    score, keep = o.select(hist, O.Params(10, 10, bins=2, l_max=2, tau=0.3))
    assert list(keep) == [O.KEEP_FIRST, O.KEEP_DROP, O.KEEP_GAP, O.KEEP_DROP]
    assert np.isclose(score[3], 0.2)


def pin_rule_causal(o):
    f = synth.generate(synth.medium().with_(width=64, height=48, frames=90))
    p = O.Params(64, 48, tau=0.05)
    h, s, k = o.run(f, p)
    for cut in (1, 2, 17, 45, 89):
        h2, s2, k2 = o.run(f[:cut], p)
        assert np.array_equal(h2, h[:cut]) and np.array_equal(k2, k[:cut]) and np.array_equal(s2, s[:cut])


def pin_hard_cuts(o):
    spec = synth.tiny_banded()
    f = synth.generate(spec)
    p = O.Params(spec.width, spec.height)
    _, score, keep = o.run(f, p)
    cuts = synth.scene_starts(spec)[1:]
    assert len(cuts) == 3
    assert (keep[cuts] == O.KEEP_NOVELTY).all(), "every hard cut between disjoint scenes is retained"
    assert (score[cuts] > 0.9).all()


def _bruteforce_mask(hist, N, tau, L):
    """The unique keep mask that satisfies the rule at every frame, found by
    checking all 2^T masks (first frame forced by the safeguard)."""
    T = len(hist)
    tau32 = np.float32(tau)
    two_n = np.float32(2 * N)
    sols = []
    for m in range(1 << T):
        mask = [(m >> t) & 1 for t in range(T)]
        ok = mask[0] == 1
        for t in range(1, T):
            if not ok:
                break
            r = max(u for u in range(t) if mask[u])
            d_adj = np.float32(np.abs(hist[t] - hist[t - 1]).sum()) / two_n
            d_ref = np.float32(np.abs(hist[t] - hist[r]).sum()) / two_n
            rule = (max(d_adj, d_ref) >= tau32) or (L > 0 and t - r >= L)
            ok = mask[t] == int(rule)
        if ok:
            sols.append(mask)
    return sols


def pin_bruteforce_4x8x8(o):
    g = _rng(16)
    hits = 0
    for trial in range(300):
        B = int(g.choice([4, 8, 32]))
        base = g.integers(0, 256, size=(8, 8, 3), dtype=np.uint8)
        frames = []
        for t in range(4):
            kind = int(g.integers(0, 3))
            if kind == 0:
                frames.append(base.copy())
            elif kind == 1:
                f = base.astype(np.int64) + g.integers(-40, 41, size=(8, 8, 3))
                frames.append(np.clip(f, 0, 255).astype(np.uint8))
            else:
                frames.append(g.integers(0, 256, size=(8, 8, 3), dtype=np.uint8))
        frames = np.stack(frames)
        tau = float(g.choice([0.05, 0.1, 0.2, 0.3, 0.5]))
        L = int(g.integers(0, 5))  # 0: no forced retention
        p = O.Params(8, 8, bins=B, l_max=L, tau=tau)
        hist_np = np.stack([np_hist(f, B) for f in frames])
        h, _, keep = o.run(frames, p)
        assert np.array_equal(h.astype(np.int64), hist_np), "4-frame histogram"
        sols = _bruteforce_mask(hist_np, 64, tau, L)
        assert len(sols) == 1, "the rule has exactly one self-consistent mask"
        assert list((keep != 0).astype(int)) == sols[0], f"trial {trial}: oracle mask differs from brute force"
        hits += sum(sols[0][1:])
    assert hits > 50, "brute force exercised too few retentions"


# ---------------------------------------------------- closing safeguards --

def pin_candidates(o):
    g = _rng(17)
    assert o.candidates(np.zeros(0, dtype=np.uint8), 4).size == 0
    for _ in range(400):
        T = int(g.integers(1, 16))
        m_min = int(g.integers(0, 9))
        keep = (g.random(T) < g.random()).astype(np.uint8) * g.integers(1, 4, size=T).astype(np.uint8)
        out = o.candidates(keep, m_min)
        base = set(np.flatnonzero(keep).tolist()) | {T - 1}
        assert list(out) == sorted(set(out.tolist())), "sorted and unique"
        assert base <= set(out.tolist()), "kept frames and the last frame are candidates"
        if len(base) >= m_min:
            assert set(out.tolist()) == base
        else:
            fill = set(np.floor(np.linspace(0, T - 1, m_min) + 0.5 + 1e-9).astype(int).tolist())
            assert set(out.tolist()) == base | fill, "uniformly spaced fill"
            assert len(out) >= min(m_min, T)


def pin_paper_defaults(o):
    with open(os.path.join(GOLDEN, "ngff_defaults.json")) as fh:
        d = json.load(fh)
    p = O.Params(1, 1)
    assert (p.bins, p.m_min, p.l_max) == (d["bins"]["value"], d["m_min"]["value"], d["l_max"]["value"])
    assert abs(p.tau - d["tau_h"]["value"]) < 1e-12


PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]


def main(path: str | None = None) -> int:
    o = O.Oracle(path) if path else O.load()
    failed = 0
    for pin in PINS:
        try:
            pin(o)
        except AssertionError as e:  # a pin caught a disagreement
            failed += 1
            print(f"FAIL {pin.__name__}: {e}")
        except Exception:  # noqa: BLE001 -- any crash counts as a failed pin
            failed += 1
            print(f"ERROR {pin.__name__}:\n{traceback.format_exc()}")
    return failed


if __name__ == "__main__":
    sys.exit(min(main(sys.argv[1] if len(sys.argv) > 1 else None), 100))
