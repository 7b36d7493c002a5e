// Slot-level OFDMA uplink that produces the completion events the release
// controller consumes (Sec. III-A, Eqs. 1-5): per slot t the eligible agents
// (payload left and t >= l_k), a causal per-resource-block choice, the bits
// each agent sends in the slot (slot length x rate), the queue update, and the
// completion slot a_k recorded once, when an agent's queue reaches zero.
// Policies (Sec. IV-B; Sec. V-A-4): max-rate, round-robin (per RB the first
// eligible agent after the previously served one, cyclically), max-weight
// (queue x rate), earliest finish (the least time to empty the queue at this
// rate) and a weighted max-rate (weight x rate: the DAG-rank and
// task-weighted variants).  Ties go to the smallest agent index.  The rates
// are an input, so the arrivals follow exactly from the channel the caller
// draws.
#include <cmath>
#include <limits>
#include <vector>

#include "rtcc.h"

extern "C" rtcc_status rtcc_uplink_simulate(int32_t n_agents, int32_t n_rb, int32_t t_max,
                                            const double* payload_bits, const int32_t* first_slot,
                                            const double* rates, double slot_s, int32_t policy,
                                            const double* weight, int32_t* completion_slot,
                                            int32_t* n_slots_used) {
  const int K = n_agents, F = n_rb;
  if (K < 1 || K > 64 || F < 1 || t_max < 1 || !payload_bits || !first_slot || !rates ||
      !completion_slot || !(slot_s > 0.0))
    return RTCC_E_ARG;
  if (policy < RTCC_SCHED_MAXRATE || policy > RTCC_SCHED_WEIGHTED) return RTCC_E_ARG;
  if (policy == RTCC_SCHED_WEIGHTED && !weight) return RTCC_E_ARG;
  const double kInf = std::numeric_limits<double>::infinity();
  std::vector<double> Q(payload_bits, payload_bits + K), d(K);
  std::vector<int> elig;
  elig.reserve(K);
  for (int k = 0; k < K; ++k) completion_slot[k] = 0;
  int rr_last = -1, done = 0, t_used = 0;
  for (int t = 1; t <= t_max && done < K; ++t) {
    t_used = t;
    const double* Rt = rates + (size_t)(t - 1) * K * F;      // [K][F] of slot t
    elig.clear();
    for (int k = 0; k < K; ++k)
      if (Q[k] > 0.0 && t >= first_slot[k]) elig.push_back(k);
    for (int k = 0; k < K; ++k) d[k] = 0.0;
    for (int f = 0; f < F && !elig.empty(); ++f) {
      int pick = -1;
      if (policy == RTCC_SCHED_ROUNDROBIN) {
        for (int step = 1; step <= K && pick < 0; ++step) {
          const int k = (rr_last + step) % K;
          for (int e : elig)
            if (e == k) {
              pick = k;
              break;
            }
        }
        rr_last = pick;
      } else {
        double best = 0.0;
        for (int k : elig) {                       // ascending k: ties keep the smaller
          const double r = Rt[(size_t)k * F + f];
          double sc;
          switch (policy) {
            case RTCC_SCHED_MAXRATE: sc = r; break;
            case RTCC_SCHED_WEIGHTED: sc = weight[k] * r; break;
            case RTCC_SCHED_MAXWEIGHT: sc = Q[k] * r; break;
            default: sc = r > 0.0 ? -Q[k] / (slot_s * r) : -kInf; break;   // earliest finish
          }
          if (pick < 0 || sc > best) {
            pick = k;
            best = sc;
          }
        }
      }
      d[pick] += slot_s * Rt[(size_t)pick * F + f];
    }
    for (int k = 0; k < K; ++k) {
      const double q_next = Q[k] - d[k] > 0.0 ? Q[k] - d[k] : 0.0;
      if (Q[k] > 0.0 && q_next == 0.0) {
        completion_slot[k] = t;
        ++done;
      }
      Q[k] = q_next;
    }
  }
  if (n_slots_used) *n_slots_used = t_used;
  return RTCC_OK;
}
