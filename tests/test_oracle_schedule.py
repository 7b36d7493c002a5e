"""Pins of the oracle's execution timeline and slot-level uplink.

The timeline is pinned by a hand-worked example (tests/golden) and by the
properties the paper states for the single-stream model: T_B - T_R = W_pre
exactly (Sec. V-C), T_R <= T_B, release causality s >= a (Eqs. 10-11), zero
gain when every encoder is still pending at the last arrival.  The uplink is
pinned by closed forms for constant rates.
"""
import json
import math
import os

import numpy as np
import pytest

import synth
from oracle import schedule as sch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "schedule_example.json")


def test_hand_worked_example():
    g = json.load(open(GOLDEN))
    for mode in ("rtcc", "barrier"):
        r = sch.simulate(g["a"], g["c_enc"], g["c_post"], mode)
        for key, val in g[mode].items():
            assert r[key] == val, (mode, key)
    r = sch.simulate(g["a"], g["c_enc"], g["c_post"], "rtcc")
    b = sch.simulate(g["a"], g["c_enc"], g["c_post"], "barrier")
    assert b["T"] - r["T"] == g["gain"]


def _rand_trace(rng, K):
    a = rng.integers(0, 50_000_000, K).tolist()
    if rng.random() < 0.3:
        a[rng.integers(0, K)] = a[0]                         # ties
    c = rng.integers(1, 8_000_000, K).tolist()
    post = rng.integers(0, 3_000_000, rng.integers(1, 4)).tolist()
    return a, c, post


def test_gain_identity_and_causality_random():
    rng = np.random.default_rng(0)
    for _ in range(3000):
        K = int(rng.integers(1, 9))
        a, c, post = _rand_trace(rng, K)
        r = sch.simulate(a, c, post, "rtcc")
        b = sch.simulate(a, c, post, "barrier")
        assert b["T"] - r["T"] == r["W_pre"]                  # Sec. V-C identity
        assert r["T"] <= b["T"]
        assert all(r["s"][k] >= a[k] for k in range(K))       # s_E >= r = a
        assert all(b["s"][k] >= max(a) for k in range(K))
        assert r["order"] == sorted(range(K), key=lambda k: (a[k], k))
        # non-overlap on the single stream
        iv = sorted(zip(r["s"], r["f"]))
        assert all(iv[j][1] <= iv[j + 1][0] for j in range(len(iv) - 1))


def test_zero_overlap_boundaries():
    c, post = [5, 6, 7], [4]
    r = sch.simulate([10, 10, 10], c, post, "rtcc")
    b = sch.simulate([10, 10, 10], c, post, "barrier")
    assert r["W_pre"] == 0 and r["T"] == b["T"] == 10 + 18 + 4
    one_r = sch.simulate([3], [9], [2], "rtcc")
    one_b = sch.simulate([3], [9], [2], "barrier")
    assert one_r == one_b


def test_well_spaced_arrivals_leave_one_encoder_in_the_tail():
    c, post = [5, 6, 7], [4, 1]
    a = [0, 100, 40]                                          # gaps >> max c
    r = sch.simulate(a, c, post, "rtcc")
    assert r["T_tail"] == c[1] + sum(post)
    b = sch.simulate(a, c, post, "barrier")
    assert b["T_tail"] == sum(c) + sum(post)


def _const_rates(T, K, F, rates):
    R = np.zeros((T, K, F))
    for k in range(K):
        R[:, k, :] = rates[k]
    return R


def test_uplink_single_agent_closed_form():
    delta, rate = 1e-3, 2.0e6
    for Bk in (1.0, 2000.0, 2001.0, 123456.0):
        R = _const_rates(500, 1, 1, [rate])
        r = sch.uplink([Bk], [1], R, delta, "maxrate")
        assert r["a"] == [math.ceil(Bk / (delta * rate))]


def test_uplink_maxrate_ties_go_to_smaller_index():
    delta, rate = 1e-3, 1.0e6
    R = _const_rates(200, 2, 1, [rate, rate])
    B = [10_500.0, 4_000.0]
    r = sch.uplink(B, [1, 1], R, delta, "maxrate")
    t0 = math.ceil(B[0] / (delta * rate))
    assert r["a"] == [t0, t0 + math.ceil(B[1] / (delta * rate))]


def test_uplink_round_robin_alternates():
    delta, rate = 1e-3, 1.0e6
    R = _const_rates(200, 2, 1, [rate, rate])
    B = [5_000.0, 5_000.0]
    r = sch.uplink(B, [1, 1], R, delta, "roundrobin")
    n = math.ceil(B[0] / (delta * rate))
    assert r["a"] == [2 * n - 1, 2 * n]
    assert r["alloc"][:4] == [[0], [1], [0], [1]]


def test_uplink_local_availability_and_infeasible():
    delta, rate = 1e-3, 1.0e6
    R = _const_rates(50, 2, 1, [rate, 2 * rate])
    r = sch.uplink([3_000.0, 3_000.0], [1, 10], R, delta, "maxrate")
    assert r["alloc"][0] == [0] and r["a"][0] == 3
    assert all(x == [-1] for x in r["alloc"][3:9])            # nobody eligible
    assert r["a"][1] == 9 + 2
    short = sch.uplink([3_000.0, 1e9], [1, 1], R, delta, "maxrate")
    assert not short["feasible"] and short["a"][1] == 0 and short["a_time"][1] == math.inf


def test_uplink_multiple_rbs_and_weights():
    delta = 1e-3
    R = np.zeros((100, 3, 2))
    R[:, 0, :] = 1.0e6
    R[:, 1, :] = 1.5e6
    R[:, 2, :] = 1.2e6
    # task weights favour agent 2 (1.2 * 1.4 > 1.5 * 1.0); both RBs go to it
    r = sch.uplink([4_000.0, 4_000.0, 4_000.0], [1, 1, 1], R, delta, "twmaxrate",
                   weight=[1.0, 1.0, 1.4])
    assert r["alloc"][0] == [2, 2]
    assert r["a"][2] == math.ceil(4_000.0 / (2 * delta * 1.2e6))
    mw = sch.uplink([10_000.0, 1_000.0, 1_000.0], [1, 1, 1], R, delta, "maxweight")
    assert mw["alloc"][0] == [0, 0]                           # largest Q * R
    er = sch.uplink([10_000.0, 1_000.0, 3_000.0], [1, 1, 1], R, delta, "earliest")
    assert er["alloc"][0] == [1, 1]                           # smallest Q / (delta R)


def test_rayleigh_rates_closed_forms():
    # R = B log2(1 + snr |h|^2): snr 3 at |h|^2 = 1 gives log2(4) = 2 bit/s/Hz,
    # snr 15 gives 4, snr 1 gives 1, and a faded-out slot (|h|^2 = 0) carries
    # nothing.  A dB/linear mix-up or a natural log fails these.
    B = 20e6
    snr = np.array([3.0, 15.0, 1.0])
    h2 = np.ones((2, 3, 4))
    h2[1, :, 1] = 0.0
    r = sch.rayleigh_rates(snr, h2, B)
    assert r.shape == (2, 3, 4)
    np.testing.assert_allclose(r[0, :, 0], [2 * B, 4 * B, B], rtol=1e-15)
    assert np.all(r[1, :, 1] == 0.0)
    # the rate doubles with |h|^2 = 5 at snr 3 (log2 16 = 4)
    assert sch.rayleigh_rates(np.array([3.0]), np.full((1, 1, 1), 5.0), B)[0, 0, 0] == \
        pytest.approx(4 * B, rel=1e-15)


def test_channel_draws_snr_is_linear_from_db():
    # Mean SNR is drawn uniform in dB over [0, 25] and returned linear: every
    # value lies in [10^0, 10^2.5] and 10 log10 of the values is uniform (mean
    # 12.5 dB); the fading power is Exp(1) (mean 1, variance 1).
    d = synth.channel_draws(4000, 50, 8, frame=0, seed=11)
    snr = d["snr"]
    assert snr.min() >= 1.0 and snr.max() <= 10 ** 2.5
    db = 10 * np.log10(snr)
    assert abs(db.mean() - 12.5) < 0.4 and abs(db.std() - 25 / math.sqrt(12)) < 0.3
    h2 = d["h2"]
    assert h2.shape == (50, 4000, 8)
    assert abs(h2.mean() - 1.0) < 0.01 and abs(h2.var() - 1.0) < 0.03
