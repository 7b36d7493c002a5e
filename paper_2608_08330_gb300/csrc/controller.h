// Release controller of RTCC (Sec. IV-C, Eqs. 17-19) -- host only.
//
// Turns validated completion events into dispatchable branches.  Each branch
// carries a state z_k (Eq. 18) and a release time r_k; the ready queue is
// ordered by (r_k, k) so simultaneous completions dispatch in index order
// (Sec. IV-C/D).  Under RTCC r_k = a_k and a branch is dispatchable as soon as
// its own event arrives; under Barrier every r_k = A = max_k a_k, so nothing is
// dispatchable until the last branch resolves.
#pragma once

#include <cstdint>
#include <vector>

#include "rtcc.h"

namespace rtcc {

class Controller {
 public:
  Controller(int n_agents, int cap_points, bool attn_ego)
      : K_(n_agents), cap_(cap_points), attn_ego_(attn_ego) {
    reset_states();
  }

  int n_agents() const { return K_; }
  rtcc_mode mode() const { return mode_; }
  bool frame_open() const { return open_; }
  bool aborted() const { return aborted_; }

  rtcc_status set_mode(rtcc_mode m);
  rtcc_status begin(uint64_t frame_id, double t0_ms);
  // Completion event e_k (Eq. 17); `out` receives dispatchable agents.
  rtcc_status complete(int agent, const void* payload, int n_points, double t_ms,
                       std::vector<int>* out);
  rtcc_status absent(int agent, double t_ms, std::vector<int>* out);
  rtcc_status mark(int agent, int state);
  rtcc_status abort();
  rtcc_status end();
  bool join_ready() const;
  bool all_resolved() const;
  rtcc_status state(int agent, int* st, double* release_ms) const;
  bool present(int agent) const { return z_[agent] != RTCC_ABSENT; }
  double last_arrival() const { return A_; }

 private:
  rtcc_status validate(int agent, double t_ms) const;
  void pop_dispatchable(std::vector<int>* out);
  void reset_states();

  int K_;
  int cap_;
  bool attn_ego_;
  rtcc_mode mode_ = RTCC_MODE_RTCC;
  bool open_ = false;
  bool aborted_ = false;
  uint64_t frame_ = 0;
  double t0_ = 0.0;
  double A_ = 0.0;
  int resolved_ = 0;
  int n_absent_ = 0;
  int z_[RTCC_MAX_AGENTS];
  double a_[RTCC_MAX_AGENTS];
  double r_[RTCC_MAX_AGENTS];
  // ready queue: released, not yet handed to the executor
  struct Entry { double r; int k; };
  std::vector<Entry> ready_;
};

}  // namespace rtcc
