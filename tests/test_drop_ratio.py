"""Eq. 9: the total drop ratio of the coarse-to-fine path composes the two
stages' ratios, D_total = 1 - (1 - D_NGFF)(1 - D_QER). Pinned to the
budget-allocation table the paper prints (tests/golden/drop_allocation.json),
whose rows split an approximately fixed total between the stages, and to the
frame counts it is computed from in the benchmark's pipeline line."""
import json
import os

REPO = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_table_rows_compose_to_their_total():
    import bench
    d = json.load(open(os.path.join(REPO, "tests", "golden", "drop_allocation.json")))
    tol = d["tolerance_pct"] / 100
    for total, ngff, qer in d["rows"]:
        T = 100_000
        m = round(T * (1 - ngff / 100))
        k = round(m * (1 - qer / 100))
        r = bench.drop_ratios(T, m, k)
        assert abs(r["total"] - total / 100) <= tol, (total, ngff, qer, r)
        assert abs(r["total"] - (1 - k / T)) < 1e-12  # the composed ratio is the fraction of frames removed


def test_edge_cases():
    import bench
    assert bench.drop_ratios(0, 0, 0) == {"ngff": 0.0, "qer": 0.0, "total": 0.0}
    r = bench.drop_ratios(3600, 127, 38)
    assert abs(r["total"] - (1 - 38 / 3600)) < 1e-12
    assert bench.drop_ratios(10, 10, 10)["total"] == 0.0
