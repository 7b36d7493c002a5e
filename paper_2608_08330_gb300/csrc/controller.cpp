// Release controller of RTCC (Sec. IV-C/D) and its standalone C ABI.
#include "controller.h"

#include <algorithm>
#include <cmath>
#include <new>

namespace rtcc {

void Controller::reset_states() {
  for (int k = 0; k < RTCC_MAX_AGENTS; ++k) {
    z_[k] = RTCC_WAITING;
    a_[k] = NAN;
    r_[k] = NAN;
  }
  ready_.clear();
  resolved_ = 0;
  n_absent_ = 0;
  A_ = 0.0;
  aborted_ = false;
}

rtcc_status Controller::set_mode(rtcc_mode m) {
  if (m != RTCC_MODE_RTCC && m != RTCC_MODE_BARRIER) return RTCC_E_ARG;
  if (open_) return RTCC_E_STATE;
  mode_ = m;
  return RTCC_OK;
}

rtcc_status Controller::begin(uint64_t frame_id, double t0_ms) {
  if (open_) return RTCC_E_STATE;
  if (!std::isfinite(t0_ms)) return RTCC_E_ARG;
  reset_states();
  open_ = true;
  frame_ = frame_id;
  t0_ = t0_ms;
  return RTCC_OK;
}

// Sec. IV-C: duplicate, premature, malformed or inconsistent events are
// rejected before any state changes.
rtcc_status Controller::validate(int agent, double t_ms) const {
  if (!open_ || aborted_) return RTCC_E_PREMATURE;
  if (agent < 0 || agent >= K_) return RTCC_E_AGENT;
  if (z_[agent] != RTCC_WAITING) return RTCC_E_DUPLICATE;
  if (!std::isfinite(t_ms)) return RTCC_E_MALFORMED;
  if (t_ms < t0_) return RTCC_E_PREMATURE;
  return RTCC_OK;
}

void Controller::pop_dispatchable(std::vector<int>* out) {
  // Under Barrier the queue only drains once every branch has resolved; then
  // r_k = A for every present branch and the (r_k, k) order is index order.
  if (mode_ == RTCC_MODE_BARRIER) {
    if (!all_resolved()) return;
    for (auto& e : ready_) {
      e.r = A_;
      r_[e.k] = A_;
    }
  }
  std::sort(ready_.begin(), ready_.end(), [](const Entry& x, const Entry& y) {
    return x.r < y.r || (x.r == y.r && x.k < y.k);
  });
  if (out) {
    for (const auto& e : ready_) out->push_back(e.k);
  }
  ready_.clear();
}

rtcc_status Controller::complete(int agent, const void* payload, int n_points, double t_ms,
                                 std::vector<int>* out) {
  rtcc_status s = validate(agent, t_ms);
  if (s != RTCC_OK) return s;
  if (n_points < 0 || n_points > cap_ || (payload == nullptr && n_points > 0))
    return RTCC_E_MALFORMED;
  z_[agent] = RTCC_RELEASED;
  a_[agent] = t_ms;
  r_[agent] = t_ms;          // release certificate, Eq. 19: r_k = a_k
  A_ = (resolved_ == 0) ? t_ms : std::max(A_, t_ms);
  ++resolved_;
  ready_.push_back({t_ms, agent});
  pop_dispatchable(out);
  return RTCC_OK;
}

rtcc_status Controller::absent(int agent, double t_ms, std::vector<int>* out) {
  rtcc_status s = validate(agent, t_ms);
  if (s != RTCC_OK) return s;
  if (attn_ego_ && agent == 0) return RTCC_E_ARG;
  if (n_absent_ + 1 >= K_) return RTCC_E_ARG;   // at least one branch present
  z_[agent] = RTCC_ABSENT;
  a_[agent] = t_ms;
  A_ = (resolved_ == 0) ? t_ms : std::max(A_, t_ms);
  ++resolved_;
  ++n_absent_;
  pop_dispatchable(out);
  return RTCC_OK;
}

rtcc_status Controller::mark(int agent, int state) {
  if (agent < 0 || agent >= K_) return RTCC_E_AGENT;
  int z = z_[agent];
  if (state == RTCC_RUNNING && z == RTCC_RELEASED) {
    z_[agent] = RTCC_RUNNING;
    return RTCC_OK;
  }
  if (state == RTCC_FINISHED && z == RTCC_RUNNING) {
    z_[agent] = RTCC_FINISHED;
    return RTCC_OK;
  }
  return RTCC_E_STATE;
}

rtcc_status Controller::abort() {
  if (!open_) return RTCC_E_STATE;
  aborted_ = true;
  ready_.clear();
  return RTCC_OK;
}

rtcc_status Controller::end() {
  if (!open_) return RTCC_E_STATE;
  open_ = false;
  return RTCC_OK;
}

bool Controller::all_resolved() const { return resolved_ == K_; }

bool Controller::join_ready() const {
  return open_ && !aborted_ && all_resolved() && n_absent_ < K_;
}

rtcc_status Controller::state(int agent, int* st, double* release_ms) const {
  if (agent < 0 || agent >= K_) return RTCC_E_AGENT;
  if (st) *st = z_[agent];
  if (release_ms) *release_ms = (z_[agent] == RTCC_WAITING || z_[agent] == RTCC_ABSENT) ? NAN : r_[agent];
  return RTCC_OK;
}

}  // namespace rtcc

// ---------------------------------------------------------------------------
// standalone C ABI
// ---------------------------------------------------------------------------

struct rtcc_controller {
  rtcc::Controller c;
  rtcc_controller(int k, int cap, bool ego) : c(k, cap, ego) {}
};

static void copy_out(const std::vector<int>& v, int32_t* released, int32_t* n_released) {
  if (n_released) *n_released = static_cast<int32_t>(v.size());
  if (released) {
    for (size_t i = 0; i < v.size(); ++i) released[i] = v[i];
  }
}

extern "C" {

rtcc_status rtcc_ctrl_create(int32_t n_agents, int32_t cap_points, int32_t attn_ego,
                             rtcc_controller** out) {
  if (!out || n_agents < 1 || n_agents > RTCC_MAX_AGENTS || cap_points < 0) return RTCC_E_ARG;
  *out = new (std::nothrow) rtcc_controller(n_agents, cap_points, attn_ego != 0);
  return *out ? RTCC_OK : RTCC_E_NOMEM;
}

void rtcc_ctrl_destroy(rtcc_controller* c) { delete c; }

rtcc_status rtcc_ctrl_set_mode(rtcc_controller* c, rtcc_mode mode) {
  return c ? c->c.set_mode(mode) : RTCC_E_ARG;
}

rtcc_status rtcc_ctrl_begin(rtcc_controller* c, uint64_t frame_id, double t0_ms) {
  return c ? c->c.begin(frame_id, t0_ms) : RTCC_E_ARG;
}

rtcc_status rtcc_ctrl_complete(rtcc_controller* c, int32_t agent, const void* payload,
                               int32_t n_points, double t_ms, int32_t* released,
                               int32_t* n_released) {
  if (!c) return RTCC_E_ARG;
  std::vector<int> v;
  rtcc_status s = c->c.complete(agent, payload, n_points, t_ms, &v);
  copy_out(v, released, n_released);
  return s;
}

rtcc_status rtcc_ctrl_absent(rtcc_controller* c, int32_t agent, double t_ms,
                             int32_t* released, int32_t* n_released) {
  if (!c) return RTCC_E_ARG;
  std::vector<int> v;
  rtcc_status s = c->c.absent(agent, t_ms, &v);
  copy_out(v, released, n_released);
  return s;
}

rtcc_status rtcc_ctrl_mark(rtcc_controller* c, int32_t agent, int32_t state) {
  return c ? c->c.mark(agent, state) : RTCC_E_ARG;
}

rtcc_status rtcc_ctrl_abort(rtcc_controller* c) { return c ? c->c.abort() : RTCC_E_ARG; }

int32_t rtcc_ctrl_join_ready(const rtcc_controller* c) { return c && c->c.join_ready() ? 1 : 0; }

rtcc_status rtcc_ctrl_state(const rtcc_controller* c, int32_t agent, int32_t* state,
                            double* release_ms) {
  return c ? c->c.state(agent, state, release_ms) : RTCC_E_ARG;
}

rtcc_status rtcc_ctrl_end(rtcc_controller* c) { return c ? c->c.end() : RTCC_E_ARG; }

}  // extern "C"
