"""Pins for the scene-change-detection + H-diff oracle (no GPU): reductions to
the histogram rule, and hand-derived keep sets on constructed histogram
sequences (ramps between two bins, holds and cuts) where every distance is an
exact dyadic fraction."""
import numpy as np
import pytest

import oracle as O
import synth
from oracle import scd_oracle as SC

N = 1024  # pixels per frame of the constructed histograms


def _hist_from_positions(pos, bins=2):
    """Histograms with pos[t] pixels in bin 1 and the rest in bin 0."""
    h = np.zeros((len(pos), bins), dtype=np.uint32)
    h[:, 1] = pos
    h[:, 0] = N - np.asarray(pos)
    return h


def _params(tau, l_max=256):
    return O.Params(32, 32, bins=2, tau=tau, l_max=l_max)  # 32 x 32 = N pixels


def _keeps(keep):
    return {int(t): int(keep[t]) for t in np.flatnonzero(keep)}


@pytest.mark.parametrize("t_cut,t_grad", [(0.30, 0.30), (0.30, 0.9), (0.45, 0.5), (2.0, 2.0)])
def test_reduces_to_histogram_rule_when_scenes_imply_novelty(t_cut, t_grad):
    """With T_b >= tau_h and T_s >= T_b no run ever opens, and every cut has
    s_adj >= T_b >= tau_h, so it is already a novelty keep: the combined rule
    must give the C oracle's histogram-rule result exactly."""
    spec = synth.medium(seed=77).with_(width=48, height=32, frames=300, mean_scene_len=9)
    fr = synth.generate(spec)
    p = O.Params(spec.width, spec.height, tau=0.30, l_max=17)
    hist, so, ko = O.load().run(fr, p)
    s2, k2 = SC.select(hist, p, t_cut, t_grad)
    assert np.array_equal(k2, ko)
    assert np.allclose(s2, so, rtol=1e-12, atol=0)  # the C oracle sums normalised bins in double


def test_two_ramps_closed_form():
    """Bin-1 counts: ramp 0, 16, .., 320 (t = 0..20), hold 320 (t = 21..23),
    ramp 336, .., 960 (t = 24..63). Every ramp step has SD = 32 / 2048 = 1/64
    (T_s = 0.01 <= SD < T_b = 1/8), a hold has SD = 0. Run 1 reaches A = 8/64
    at t = 8 (scene), the hold ends it, run 2 reaches 8/64 at t = 24 + 7 = 31
    (scene); s_ref from r = 31 (count 448) reaches 512/1024 = tau = 0.5 at
    count 960, t = 63 (novelty). No other keep: A passes T_b only once per run."""
    pos = [16 * t for t in range(21)] + [320] * 3 + [320 + 16 * (t - 23) for t in range(24, 64)]
    h = _hist_from_positions(pos)
    _, keep = SC.select(h, _params(0.5), 0.125, 0.01)
    assert _keeps(keep) == {0: 3, 8: SC.KEEP_SCENE, 31: SC.KEEP_SCENE, 63: O.KEEP_NOVELTY}


def test_cut_resets_the_run():
    """Five ramp steps (A = 5/64), a cut of 128 pixels (SD = 1/8 = T_b: a scene
    change that also ends the run), five more ramp steps: A restarts from 0
    and stays below T_b, so the cut is the only scene change."""
    pos = [16 * t for t in range(6)] + [208] + [208 + 16 * i for i in range(1, 6)]
    h = _hist_from_positions(pos)
    _, keep = SC.select(h, _params(1.5), 0.125, 0.01)
    assert _keeps(keep) == {0: 3, 6: SC.KEEP_SCENE}


def test_hold_resets_the_run_and_low_steps_never_accumulate():
    """Steps of 4 pixels (SD = 1/256 < T_s) never join a run; a run of four
    1/64 steps, a hold and four more never reaches 8/64."""
    pos = [4 * t for t in range(30)]
    _, keep = SC.select(_hist_from_positions(pos), _params(1.5), 0.125, 0.01)
    assert _keeps(keep) == {0: 3}
    pos = [16 * t for t in range(5)] + [64] + [64 + 16 * i for i in range(1, 5)]
    _, keep = SC.select(_hist_from_positions(pos), _params(1.5), 0.125, 0.01)
    assert _keeps(keep) == {0: 3}


@pytest.mark.parametrize("tau,code", [(1.5, SC.KEEP_SCENE), (0.3, O.KEEP_NOVELTY)])
def test_hard_cut_code_precedence(tau, code):
    """A cut between disjoint histograms (SD = 1): a scene change, reported as
    novelty when s >= tau_h also holds (novelty first)."""
    pos = [0] * 10 + [N] * 10
    _, keep = SC.select(_hist_from_positions(pos), _params(tau), 0.30, 0.10)
    assert _keeps(keep) == {0: 3, 10: code}


def test_scene_change_beats_gap_and_restarts_it():
    """Constant frames with L_max = 4 are kept at 4, 8, ... by the gap rule; a
    cut at t = 4 coincides with a gap keep and is reported as a scene change;
    a cut at t = 10 restarts the gap count (next gap keep at 14, not 12)."""
    pos = [0] * 4 + [N] * 6 + [0] * 10
    _, keep = SC.select(_hist_from_positions(pos), _params(1.5, l_max=4), 0.30, 0.10)
    assert _keeps(keep) == {0: 3, 4: SC.KEEP_SCENE, 8: O.KEEP_GAP, 10: SC.KEEP_SCENE, 14: O.KEEP_GAP,
                            18: O.KEEP_GAP}


def test_prefix_causality_and_twin_comparison_state():
    spec = synth.medium(seed=78).with_(width=40, height=24, frames=240, mean_scene_len=6)
    fr = synth.generate(spec)
    p = O.Params(spec.width, spec.height, tau=0.35, l_max=23)
    hist = np.stack([O.load().histogram(f, p) for f in fr])
    s, k = SC.select(hist, p, 0.2, 0.03)
    assert (k == SC.KEEP_SCENE).any() and (k == O.KEEP_NOVELTY).any()
    for cut in (1, 2, 57, 150):
        s2, k2 = SC.select(hist[:cut], p, 0.2, 0.03)
        assert np.array_equal(k2, k[:cut]) and np.array_equal(s2, s[:cut])
    # the run state carried across a split equals the single pass
    adj = [0] + [SC.l1(hist[t], hist[t - 1]) for t in range(1, len(hist))]
    f_all, a_all = SC.scene_changes(adj, 2 * p.npix, 0.2, 0.03)
    f1, a1 = SC.scene_changes(adj[:100], 2 * p.npix, 0.2, 0.03)
    f2, a2 = SC.scene_changes([0] + adj[100:], 2 * p.npix, 0.2, 0.03, acc0=a1)
    assert np.array_equal(np.concatenate([f1, f2[1:]]), f_all) and a2 == a_all
