"""The gain model bench.py uses for its predicted-vs-measured check agrees
with the oracle's single-stream timeline (Eqs. 20-22): T_B - T_R, which is
also the pre-arrival encoder work W_pre."""
import numpy as np

import bench
from oracle import schedule as sch


def test_predicted_gain_matches_the_timeline_oracle():
    rng = np.random.default_rng(0)
    for _ in range(500):
        K = int(rng.integers(1, 9))
        a = [int(x) for x in rng.integers(0, 400, size=K)]
        c = [int(x) for x in rng.integers(1, 200, size=K)]
        cp = int(rng.integers(0, 100))
        r = sch.simulate(a, c, [cp], "rtcc")
        b = sch.simulate(a, c, [cp], "barrier")
        g = bench.predicted_gain(a, c, cp)
        assert g == b["T"] - r["T"] == r["W_pre"]


def test_controller_decision_timing_runs_without_gpu():
    from paper_2608_08330_gb300 import rtcc as R
    R.load()
    cc = R.rtcc_ctrl_create(6, 1000)
    for f in range(3):
        assert R.rtcc_ctrl_begin(cc, f + 1, 0.0) == R.OK
        for k in range(6):
            s, rel = R.rtcc_ctrl_complete(cc, k, True, 10, float(k))
            assert s == R.OK and rel == [k]
        for k in range(6):
            assert R.rtcc_ctrl_mark(cc, k, R.RUNNING) == R.OK
            assert R.rtcc_ctrl_mark(cc, k, R.FINISHED) == R.OK
        assert R.rtcc_ctrl_end(cc) == R.OK
    R.rtcc_ctrl_destroy(cc)


def test_paired_gain_bootstrap():
    rng = np.random.default_rng(3)
    t_r = rng.uniform(0.1, 0.2, 40)
    t_b = t_r + 0.2 + rng.normal(0, 0.01, 40)
    g = bench.paired_gain(t_b, t_r)
    assert g["pairs"] == 40 and g["positive"] == 40
    assert abs(g["mean_ms"] - float(np.mean(t_b - t_r))) < 1e-12
    lo, hi = g["ci95_ms"]
    assert lo < g["mean_ms"] < hi and hi - lo < 0.02
    assert g == bench.paired_gain(t_b, t_r)                      # seeded
    assert bench.paired_gain([], []) is None
    one = bench.paired_gain([0.3], [0.1])
    assert one["ci95_ms"][0] == one["ci95_ms"][1] == one["mean_ms"]
