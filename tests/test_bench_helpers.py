"""The host-side helpers that turn a run into bench.py's JSON line: the
oracle parity block (keep codes, score error, the tolerance band around
tau_h) and the per-config summaries. Plain numpy on the CPU."""
import numpy as np
import pytest

import bench


def test_parity_block_equal_run():
    so = np.array([0.0, 0.5, 0.25, 0.75])  # exact in fp32
    ko = np.array([3, 1, 0, 1], dtype=np.uint8)
    d = bench.parity_block(0.30, so.astype(np.float32), ko, so, ko, hist=np.ones((4, 2)), want_hist=np.ones((4, 2)),
                           idx=np.array([0, 1, 3]), want_idx=np.array([0, 1, 3]))
    assert d["keep_equal"] and d["hist_equal"] and d["candidates_equal"]
    assert d["keep_mismatch_outside_band"] == 0 and d["band_frames"] == [] and d["band_count"] == 0
    assert d["max_rel_score_err"] == 0.0  # 0.0 against 0.0 counts as equal
    assert d["frames"] == 4


def test_parity_block_band_and_mismatches():
    tau = 0.30
    so = np.array([tau, tau * (1 + 5e-7), tau * (1 - 2e-6), 0.7, 0.0])
    sg = so.copy()
    sg[3] = 0.7 * (1 + 3e-6)  # a score error above the tolerance
    ko = np.array([1, 1, 0, 1, 0], dtype=np.uint8)
    kg = ko.copy()
    kg[0] = 0  # a decision flipped inside the band
    d = bench.parity_block(tau, sg, kg, so, ko)
    assert d["band_frames"] == [0, 1] and d["band_count"] == 2  # |s - tau| <= 1e-6 tau; frame 2 is outside
    assert not d["keep_equal"] and d["keep_mismatch_outside_band"] == 0
    assert d["max_rel_score_err"] == pytest.approx(3e-6, rel=1e-3)
    kg[3] = 0  # and one outside it
    assert bench.parity_block(tau, sg, kg, so, ko)["keep_mismatch_outside_band"] == 1
    sg[4] = 1e-3  # a nonzero score where the oracle has zero is an error, not a division by zero
    assert bench.parity_block(tau, sg, ko, so, ko)["max_rel_score_err"] > 1.0


def test_parity_block_reports_unequal_histograms_and_candidates():
    d = bench.parity_block(0.3, [0.1], [0], [0.1], [0], hist=np.array([[1, 2]]), want_hist=np.array([[1, 3]]),
                           idx=np.array([0, 2]), want_idx=np.array([0, 1]))
    assert d["hist_equal"] is False and d["candidates_equal"] is False
    assert bench.parity_block(0.3, [0.1], [0], [0.1], [0], want_hist=np.zeros(2))["hist_equal"] is False


def test_compact_rounds_floats_only():
    x = {"a": 1.23456789, "b": [2.0000049, 7], "c": "text", "d": {"e": 123456.789}}
    assert bench._compact(x, 3) == {"a": 1.23, "b": [2.0, 7], "c": "text", "d": {"e": 123000.0}}


def test_rare_event_summary_collects_recall_and_parity_over_taus():
    def par(equal, err, band):
        return {"keep_equal": equal, "max_rel_score_err": err, "band_frames": band, "band_count": len(band)}
    d = {"workload": "w", "frames_per_s": 2.5e6, "events": 40, "seconds": 1.0,
         "taus": {"0.3": {"keep_ratio": 0.1, "event_frame_recall": 0.2, "event_recall": 0.4, "parity": par(True, 1e-8, [])},
                  "0.1": {"keep_ratio": 0.3, "event_frame_recall": 0.6, "event_recall": 0.9,
                          "parity": par(False, 4e-8, [17, 3])}}}
    s = bench._config_summary("rare_event", d)
    assert s["recall_by_tau"] == {"0.3": [0.1, 0.2, 0.4], "0.1": [0.3, 0.6, 0.9]}
    assert s["recall_fields"] == ["keep_ratio", "event_frame_recall", "event_recall"]
    assert s["parity"] == {"keep_equal_every_tau": False, "max_rel_score_err": 4e-8, "band_frames": [3, 17]}
    assert "taus" not in s and s["seconds"] == 1.0


def test_config_summary_keeps_the_parity_verdict():
    d = {"workload": "w", "pipelined_frames_per_s": 1.0e6, "latency_ms_p50": 0.0195,
         "e2e": {"frames_per_s": 2.7e5, "how": "long text"},
         "parity": {"frames": 600, "keep_equal": False, "keep_mismatch_outside_band": 0, "band_frames": [5],
                    "band_count": 1, "score_rtol": 1e-6, "max_rel_score_err": 5e-8, "candidates_equal": True}}
    s = bench._config_summary("medium", d)
    assert s["e2e"] == {"frames_per_s": 2.7e5}
    assert s["parity"] == {"frames": 600, "keep_equal": False, "keep_mismatch_outside_band": 0, "band_frames": [5],
                           "max_rel_score_err": 5e-8, "candidates_equal": True}
