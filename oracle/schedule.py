"""Execution-timeline and uplink models of RTCC (oracle).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Two parts, both written from the paper's definitions:

* :func:`simulate` -- the single non-preemptive, work-conserving GPU stream of
  Sec. III-B (Eqs. 8-10) under a release rule (Eq. 11).  RTCC follows Eqs.
  20-22 (encoders dispatched in (a_k, k) order, each starting at
  max(a_sigma(j), g_{j-1})); Barrier releases every encoder at A = max_k a_k
  (Sec. V, opening paragraph) in index order.  The post-join subgraph runs
  after the last encoder in topological order (Sec. IV-D).  T and T_tail are
  Eqs. 12-13.  Times are integers (e.g. ns) so the identity
  T_B - T_R = W_pre reported in Sec. V-C holds exactly.

* :func:`uplink` -- the slot-level OFDMA uplink of Sec. III-A (Eqs. 1-5) with a
  pluggable causal RB policy (Sec. IV-B, Eqs. 15-17; Sec. IV-E, Eqs. 23-25;
  Sec. V-A-3, Eqs. 27-28): eligible set at the start of each slot, per-RB
  argmax with ties to the smallest index, slot payload, queue evolution, and
  the completion slot, recorded once per agent on the transition of its queue
  to zero.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence

import numpy as np

INF = float("inf")


def simulate(a: Sequence[int], c_enc: Sequence[int], c_post: Sequence[int],
             mode: str) -> Dict[str, object]:
    """Timeline of one frame under the single-stream GPU model.

    a      -- per-agent arrival (= release under RTCC) times, integers.
    c_enc  -- per-agent encoder service times c_{E_k}.
    c_post -- service times of the post-join nodes, in topological order.
    mode   -- "rtcc" or "barrier".

    Returns order (dispatch order), s and f (per-agent encoder start/finish,
    indexed by agent), A, T (= f_o), T_tail = T - A, and W_pre = the encoder
    busy time inside [0, A) (the pre-arrival encoder work).
    """
    K = len(a)
    A = max(a)
    if mode == "rtcc":
        order = sorted(range(K), key=lambda k: (a[k], k))
        release = list(a)
    elif mode == "barrier":
        order = list(range(K))
        release = [A] * K
    else:
        raise ValueError(mode)
    s = [0] * K
    f = [0] * K
    g = 0
    for k in order:
        s[k] = max(release[k], g)
        f[k] = s[k] + c_enc[k]
        g = f[k]
    t = g
    for c in c_post:
        t = t + c
    w_pre = 0
    for k in range(K):
        w_pre += max(0, min(f[k], A) - min(s[k], A))
    return {"order": order, "s": s, "f": f, "A": A, "T": t, "T_tail": t - A,
            "W_pre": w_pre}


# --------------------------------------------------------------------------
# slot-level uplink
# --------------------------------------------------------------------------

POLICIES = ("maxrate", "roundrobin", "maxweight", "earliest", "dagrank", "twmaxrate")


def uplink(B: Sequence[float], ell: Sequence[int], R: np.ndarray, delta: float,
           policy: str, weight: Optional[Sequence[float]] = None) -> Dict[str, object]:
    """Arrival vector of one frame from per-slot rates and a causal policy.

    B      -- payload sizes B_k (bits).
    ell    -- earliest transmission slot l_k (slots are 1-based).
    R      -- rates R_{k,f}[t] (bit/s), shape [T_max][K][F]; slot t is R[t-1].
    delta  -- slot duration (s).
    policy -- "maxrate" (score R), "twmaxrate" / "dagrank" (score w_k R with
              weight = q or omega), "maxweight" (Q_k R), "earliest"
              (-Q_k / (delta R), the negative time to finish at this rate), or
              "roundrobin": per RB, the first eligible agent after the
              previously served one in cyclic index order.
    Ties go to the smallest agent index.

    Returns a (completion slot index t per agent, 0 for "never"), a_time
    (= t * delta, inf for never), feasible (all delivered), and the slot-by-slot
    allocation x [T_used][F] (agent index or -1).
    """
    T_max, K, F = R.shape
    Q = [float(b) for b in B]
    comp = [0] * K
    rr_last = -1
    alloc: List[List[int]] = []
    for t in range(1, T_max + 1):
        Rt = R[t - 1]
        elig = [k for k in range(K) if Q[k] > 0.0 and t >= ell[k]]
        x = [-1] * F
        for f in range(F):
            if not elig:
                continue
            if policy == "roundrobin":
                pick = None
                for step in range(1, K + 1):
                    k = (rr_last + step) % K
                    if k in elig:
                        pick = k
                        break
                rr_last = pick
                x[f] = pick
                continue
            best = None
            best_score = None
            for k in elig:                      # ascending k: ties keep the smaller
                r = float(Rt[k, f])
                if policy == "maxrate":
                    sc = r
                elif policy in ("twmaxrate", "dagrank"):
                    sc = float(weight[k]) * r
                elif policy == "maxweight":
                    sc = Q[k] * r
                elif policy == "earliest":
                    sc = -Q[k] / (delta * r) if r > 0.0 else -INF
                else:
                    raise ValueError(policy)
                if best is None or sc > best_score:
                    best, best_score = k, sc
            x[f] = best
        alloc.append(x)
        d = [0.0] * K
        for f in range(F):
            if x[f] >= 0:
                d[x[f]] += delta * float(Rt[x[f], f])
        for k in range(K):
            q_next = max(0.0, Q[k] - d[k])
            if Q[k] > 0.0 and q_next == 0.0:
                comp[k] = t
            Q[k] = q_next
        if all(c > 0 for c in comp):
            break
    a_time = [c * delta if c > 0 else INF for c in comp]
    return {"a": comp, "a_time": a_time, "feasible": all(c > 0 for c in comp),
            "alloc": alloc}


def rayleigh_rates(snr: np.ndarray, h2: np.ndarray, bandwidth: float) -> np.ndarray:
    """R_{k,f}[t] = bandwidth * log2(1 + snr_k |h|^2), shape of h2 ([T][K][F]).

    The per-RB Shannon rate of a Rayleigh-faded link with mean SNR snr_k.  Sec.
    III-A leaves the rate model open (loss, fading and blockage are all
    allowed); this is the model of the 4-agent uplink-sweep workload.
    """
    return bandwidth * np.log2(1.0 + snr[None, :, None] * h2)
