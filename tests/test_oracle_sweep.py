"""The measured-DAG sweep of Sec. V-D, reduced for the CPU suite.

Six agents (the paper's six branches) share an F = 8 resource-block OFDMA
uplink with Rayleigh fading; five causal schedulers (Eq. of Sec. V-A-4:
MaxRate, MaxWeight, EarliestRelease, DAGRank with normalised upward ranks,
Task-Weighted MaxRate with the paper's fixed q) turn each channel trace into
a branch-arrival vector; the single-stream timeline then gives T_R and T_B
with the paper's profiled service times (six encoders 55.98 ms in all, the
fusion/task subgraph 16.76 ms; Sec. V-E).  Over 4 payload scales x 5
bandwidth scales x 5 schedulers x 30 traces (the paper's 3,000 trials) every
feasible trial must satisfy T_B - T_R = W_pre exactly and T_R <= T_B, and
RTCC must gain in most of them (the paper: 2,984 of 3,000, the rest at
zero-overlap boundaries).  The payload and bandwidth scales, F = 8 and the
normalised upward rank are our readings of Sec. V-D.
"""
import numpy as np

import synth
from oracle import schedule as sch

K, F = 6, 8
DELTA = 1e-3                                   # slot, s
Q = [1.00, 0.80, 1.20, 0.70, 1.05, 0.60]       # task weights (Sec. V-A-4)
C_ENC = [9_330_000] * K                        # ns; 55.98 ms over six encoders
C_POST = [16_760_000]                          # ns
GAMMAS = (0.25, 0.5, 1.0, 2.0)                 # payload = gamma x 16 B x 100,000 points
BETAS = (0.5, 0.75, 1.0, 1.5, 2.0)             # bandwidth = beta x 20 MHz over F RBs
POLICIES = ("maxrate", "maxweight", "earliest", "dagrank", "twmaxrate")


def _omega():
    rank = [c + C_POST[0] for c in C_ENC]      # upward rank: encoder + the post-join after it
    return [r / max(rank) for r in rank]


def _trial(gamma, beta, pol, frame, omega):
    """(T_R, T_B, W_pre) in ns of one trace and scheduler; None if infeasible."""
    d = synth.channel_draws(K, 4000, F, frame=frame, seed=5)
    rates = sch.rayleigh_rates(d["snr"], d["h2"], beta * 20e6 / F)
    w = Q if pol == "twmaxrate" else omega if pol == "dagrank" else None
    up = sch.uplink([gamma * 16 * 100_000 * 8] * K, [1] * K, rates, DELTA, pol, weight=w)
    if not up["feasible"]:
        return None
    a = [int(t) * 1_000_000 for t in up["a"]]                  # slot index -> ns
    r = sch.simulate(a, C_ENC, C_POST, "rtcc")
    b = sch.simulate(a, C_ENC, C_POST, "barrier")
    return r["T"], b["T"], r["W_pre"]


def test_sweep_keeps_the_gain_identity():
    traces = 30
    omega = _omega()
    n_ok = n_pos = 0
    for ci, (gamma, beta) in enumerate((g, b) for g in GAMMAS for b in BETAS):
        for tr in range(traces):
            for pol in POLICIES:
                res = _trial(gamma, beta, pol, 1000 * ci + tr, omega)
                if res is None:
                    continue
                t_r, t_b, w_pre = res
                assert t_b - t_r == w_pre, (gamma, beta, pol, tr)
                assert t_r <= t_b
                n_ok += 1
                n_pos += t_b > t_r
    # heavy payloads on narrow bands may not finish within 4000 slots
    assert n_ok >= 0.9 * len(GAMMAS) * len(BETAS) * len(POLICIES) * traces
    assert n_pos >= 0.95 * n_ok                # gains vanish only at zero-overlap boundaries
