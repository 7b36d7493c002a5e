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


def test_gap_compression_leaves_both_tails_unchanged():
    # The bench replays arrival traces with long inter-arrival gaps shortened
    # to a cap.  On the single-stream timeline (Eqs. 20-22) neither mode's
    # tail T - A changes while the cap is at least the encoder work that can
    # be queued when a gap begins (here: the sum of all service times).
    rng = np.random.default_rng(5)
    for _ in range(500):
        K = int(rng.integers(1, 9))
        c = [int(x) for x in rng.integers(1, 300, size=K)]
        cp = int(rng.integers(0, 100))
        a = [int(x) for x in rng.integers(0, 20_000, size=K)]
        cap = sum(c) + int(rng.integers(0, 50))
        t = [int(round(x)) for x in bench.compress_gaps(a, float(cap))]
        for mode in ("rtcc", "barrier"):
            assert sch.simulate(t, c, [cp], mode)["T_tail"] == sch.simulate(a, c, [cp], mode)["T_tail"]
        # order kept, no gap longer than the cap, the first arrival at 0
        order = sorted(range(K), key=lambda k: (a[k], k))
        assert t[order[0]] == 0
        assert all(0 <= t[order[j]] - t[order[j - 1]] <= cap for j in range(1, K))
        assert sorted(range(K), key=lambda k: (t[k], k)) == order


def test_gap_compression_below_the_queued_work_can_change_the_tail():
    # the condition matters: one branch of 100 still running when the next
    # arrives 10 later delays it, but not if the gap is cut to 1 below the
    # 100 of queued work (the RTCC tail grows), so the cap must cover it
    a, c = [0, 150], [100, 100]
    full = sch.simulate(a, c, [10], "rtcc")["T_tail"]
    cut = sch.simulate([int(x) for x in bench.compress_gaps(a, 99.0)], c, [10], "rtcc")["T_tail"]
    assert full == 110 and cut == 111
