"""Pins for the alternative-signal oracle (low-res difference, dHash), no GPU."""
import numpy as np
import pytest

import oracle as O
from oracle import signals_oracle as SO


def _gray(values_hw):
    v = np.asarray(values_hw, dtype=np.uint8)
    return np.repeat(v[..., None], 3, axis=-1)


def test_cell_sums_brute_force():
    g = np.random.default_rng(1)
    for (H, W) in ((8, 9), (17, 23), (32, 48)):
        p = O.Params(W, H)
        f = g.integers(0, 256, size=(H, W, 3), dtype=np.uint8)
        y = O.load().luma_map(f, p).astype(np.int64)
        for grid in ((16, 16), (8, 9)):
            if H < grid[0] or W < grid[1]:
                continue
            S, n = SO.cell_sums(f, p, grid)
            S2 = np.zeros(grid, dtype=np.int64)
            n2 = np.zeros(grid, dtype=np.int64)
            for yy in range(H):
                for xx in range(W):
                    S2[yy * grid[0] // H, xx * grid[1] // W] += y[yy, xx]
                    n2[yy * grid[0] // H, xx * grid[1] // W] += 1
            assert np.array_equal(S, S2) and np.array_equal(n, n2)
            assert S.sum() == y.sum() and n.sum() == H * W


def test_dhash_of_gradients():
    H, W = 32, 72
    p = O.Params(W, H)
    ramp = np.tile(np.arange(W) * 3, (H, 1))
    up = SO.features(_gray(ramp), p, SO.DHASH)
    down = SO.features(_gray(ramp[:, ::-1]), p, SO.DHASH)
    assert up.sum() == 0, "brighter to the right: no bit set"
    assert down.sum() == 64, "darker to the right: every bit set"
    assert SO.numerator(up, down, SO.DHASH) / SO.denominator(p, SO.DHASH) == 1.0


def test_brightness_shift_closed_forms():
    g = np.random.default_rng(2)
    H, W = 48, 64
    p = O.Params(W, H)
    base = g.integers(20, 200, size=(H, W))
    for delta in (1, 7, 40):
        a, b = _gray(base), _gray(base + delta)
        fa, fb = SO.features(a, p, SO.LOWRES), SO.features(b, p, SO.LOWRES)
        assert SO.numerator(fa, fb, SO.LOWRES) == delta * H * W  # d = delta / 255 exactly
        ha, hb = SO.features(a, p, SO.DHASH), SO.features(b, p, SO.DHASH)
        assert SO.numerator(ha, hb, SO.DHASH) == 0, "a uniform shift keeps every left/right order"
    assert SO.numerator(fa, fa, SO.LOWRES) == 0


@pytest.mark.parametrize("kind", [SO.LOWRES, SO.DHASH])
def test_rule_special_cases(kind):
    g = np.random.default_rng(3)
    T, H, W = 40, 32, 36
    frames = g.integers(0, 256, size=(T, H, W, 3), dtype=np.uint8)
    for L in (1, 5, 30):
        _, _, keep = SO.run(frames, O.Params(W, H, l_max=L, tau=0.0), kind)
        assert keep[0] == O.KEEP_FIRST and (keep[1:] == O.KEEP_NOVELTY).all()
        _, _, keep = SO.run(frames, O.Params(W, H, l_max=L, tau=1.5), kind)
        assert list(np.flatnonzero(keep)) == list(range(0, T, L))
    _, _, keep = SO.run(frames, O.Params(W, H, l_max=0, tau=1.5), kind)
    assert list(np.flatnonzero(keep)) == [0], "L_max = 0: no forced retention"
    f, s, k = SO.run(frames, O.Params(W, H, tau=0.2), kind)
    for cut in (1, 9, 25):
        f2, s2, k2 = SO.run(frames[:cut], O.Params(W, H, tau=0.2), kind)
        assert np.array_equal(k2, k[:cut]) and np.array_equal(s2, s[:cut])


def test_flat_frames_closed_forms():
    """A flat frame has equal cell means everywhere: no dHash bit is set
    (strict comparison), even where cells hold different pixel counts
    (64 x 48 over 9 columns: 7 or 8 pixels). Black against white is the
    largest low-res difference: d = 255 W H / (255 W H) = 1."""
    H, W = 48, 64
    p = O.Params(W, H)
    for v in (0, 37, 255):
        assert SO.features(_gray(np.full((H, W), v)), p, SO.DHASH).sum() == 0
    black, white = _gray(np.zeros((H, W))), _gray(np.full((H, W), 255))
    fa, fb = SO.features(black, p, SO.LOWRES), SO.features(white, p, SO.LOWRES)
    assert SO.numerator(fa, fb, SO.LOWRES) / SO.denominator(p, SO.LOWRES) == 1.0


def _hashes(*bit_sets):
    """dHash feature rows with the given bits set."""
    f = np.zeros((len(bit_sets), 64), dtype=np.int64)
    for i, bits in enumerate(bit_sets):
        f[i, list(bits)] = 1
    return f


def test_rule_terms_on_constructed_hashes():
    """Only the adjacent term crosses tau: X and Y each differ from the
    reference A in 16 bits (d = 0.25) and from each other in 32 (d = 0.5).
    Only the reference term crosses: a drift of 8 bits per frame (adjacent
    d = 0.125) reaches 24 bits from the reference (0.375) at frame 3, kept
    also at tau = 0.375 (s >= tau, Eq. 5)."""
    p = O.Params(16, 16, tau=0.4, l_max=100)
    _, keep = SO.select(_hashes([], range(16), range(16, 32)), p, SO.DHASH)
    assert list(keep) == [O.KEEP_FIRST, O.KEEP_DROP, O.KEEP_NOVELTY]
    for tau in (0.3, 0.375):
        p = O.Params(16, 16, tau=tau, l_max=100)
        score, keep = SO.select(_hashes([], range(8), range(16), range(24), range(32)), p, SO.DHASH)
        assert list(keep) == [O.KEEP_FIRST, O.KEEP_DROP, O.KEEP_DROP, O.KEEP_NOVELTY, O.KEEP_DROP]
        assert list(score[1:]) == [0.125, 0.25, 0.375, 0.125]
