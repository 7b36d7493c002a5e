"""The library's slot-level uplink (rtcc_uplink_simulate, host code) against
the oracle's (Sec. III-A, Eqs. 1-5): the same rates must give the same
completion slot for every agent, for every policy, bit for bit (both sides
subtract the same float64 slot payloads in the same order)."""
import numpy as np
import pytest

import synth
from oracle import schedule as sch
from paper_2608_08330_gb300 import build as B

POLICIES = [("maxrate", 0), ("roundrobin", 1), ("maxweight", 2), ("earliest", 3), ("dagrank", 4)]


@pytest.fixture(scope="module")
def R():
    B.build()
    from paper_2608_08330_gb300 import rtcc
    rtcc.load()
    return rtcc


@pytest.mark.parametrize("name,code", POLICIES)
@pytest.mark.parametrize("K,F,gamma", [(4, 1, 0.25), (4, 1, 2.0), (6, 8, 1.0), (3, 2, 0.5)])
def test_uplink_matches_oracle(R, name, code, K, F, gamma):
    T = 1500
    for frame in range(6):
        d = synth.channel_draws(K, T, F, frame=frame, seed=13)
        rates = sch.rayleigh_rates(d["snr"], d["h2"], 20e6 / F)
        rng = np.random.default_rng([frame, K, F])
        bits = gamma * 16 * 8 * rng.integers(20_000, 100_000, K).astype(np.float64)
        ell = rng.integers(1, 6, K)
        wt = rng.uniform(0.2, 1.0, K)
        want = sch.uplink(bits, ell, rates, 1e-3, name, weight=wt)
        got, used = R.rtcc_uplink_simulate(bits, ell, rates, 1e-3, code, weight=wt)
        assert got.tolist() == list(want["a"]), (name, frame)
        assert used == (max(want["a"]) if want["feasible"] else T)


def test_uplink_rejects_bad_arguments(R):
    r = np.ones((4, 2, 1))
    with pytest.raises(R.RTCCError):
        R.rtcc_uplink_simulate([1.0, 1.0], [1, 1], r, 0.0, 0)           # slot length 0
    with pytest.raises(R.RTCCError):
        R.rtcc_uplink_simulate([1.0, 1.0], [1, 1], r, 1e-3, 9)          # unknown policy
    with pytest.raises(R.RTCCError):
        R.rtcc_uplink_simulate([1.0, 1.0], [1, 1], r, 1e-3, 4)          # weights missing
