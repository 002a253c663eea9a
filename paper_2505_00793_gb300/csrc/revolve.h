// Binomial checkpoint schedule for the reverse sweep (host code).
//
// Section 4 names binomial checkpointing (Griewank's "revolve") as the way to cut the static
// memory of the theta_t store below the T + 1 parameter copies of per-step checkpointing.
// The sweep reverses inner steps t = T-1, ..., 0 and needs the state S_t = (theta_t and the
// optimiser state m_t, v_t) when it reverses step t.  With s snapshot slots besides S_0, a
// schedule stores some states and recomputes the others by re-running inner steps forward
// from a stored one.  This file computes the schedule that re-runs the fewest inner steps.
// The classical recursion over split points defines the optimum:
//
//   F(n, s)  forward steps needed to reverse n consecutive steps [i, i + n) when S_i is
//            stored and s slots are free:  F(1, s) = 0,  F(n, 0) = n (n - 1) / 2 (every S_t
//            recomputed from S_i), and for s > 0
//            F(n, s) = min(F(n, s - 1), min_{0<m<n} m + F(n - m, s - 1) + F(m, s)):
//            advance m steps, keep S_{i+m} in a slot, reverse the right part with one slot
//            fewer, free the slot and reverse the left part.
//   G(n, s)  the same for the top level, where the rollout has already run through the
//            segment and can leave S_{i+m} in a slot on its way (no extra forward steps):
//            G(1, s) = 0,  G(n, 0) = n (n - 1) / 2,
//            G(n, s) = min(G(n, s - 1), min_{0<m<n} G(n - m, s - 1) + F(m, s)).
//
// Both have closed forms through Griewank's minimal count t(l, c) = r l - C(c + r, c + 1) for
// reversing l steps with c checkpoints (r the least integer with C(c + r, c) >= l, Griewank
// 1992):  F(n, s) = t(n, s + 1)  and  G(n, s) = t(n + 1, s + 1) - n.  The builder walks the
// recursion and takes, at each node, the fewest slots and then the smallest split m that
// reach the closed-form value, so the schedule needs no O(T^2 s) table: building one costs
// O(T) nodes, each scanning its splits.
//
// Slots: 0 holds S_0; 1..s are the snapshot slots; s + 1 and s + 2 are two scratch slots
// that an advance ping-pongs through, ending in its destination (S_T after the rollout and
// states recomputed only to be reversed at once live there).  The schedule is a list of
// actions after the initial rollout; the rollout itself leaves S_t in slot `keep[t]` for the
// split points of the top-level recursion.
#pragma once

#include <stdint.h>

#include <vector>

namespace mf {

struct RevolveAct {
  enum Kind { ADV = 0, REV = 1 } kind;
  int t0 = 0, t1 = 0;   // ADV: S_t0 -> S_t1;  REV: step t0
  int src = 0;          // ADV: slot of S_t0;  REV: slot of S_t0
  int dst = 0;          // ADV: slot that receives S_t1
};

struct RevolveSchedule {
  int T = 0, s = 0;
  std::vector<int> keep;            // [T + 1]: slot the rollout leaves S_t in, or -1
  int slot_T = 0;                   // slot of S_T after the rollout
  std::vector<RevolveAct> acts;     // after the rollout and the outer gradient
  int64_t recompute = 0;            // inner steps re-run by the sweep: G(T, s)
  int n_slots() const { return s + 3; }
  int scratch(int j) const { return s + 1 + j; }
};

namespace revolve_detail {

// Griewank's t(l, c): forward steps to reverse l steps with c >= 1 checkpoints.
inline int64_t griewank_t(int64_t l, int64_t c) {
  if (l <= 1) return 0;
  if (c == 1) return l * (l - 1) / 2;
  int64_t r = 0, b = 1;                 // b = C(c + r, c)
  while (b < l) { ++r; b = b * (c + r) / r; }
  return r * l - b * r / (c + 1);       // C(c + r, c + 1) = C(c + r, c) r / (c + 1)
}

inline int64_t F(int n, int s) { return griewank_t(n, static_cast<int64_t>(s) + 1); }
inline int64_t G(int n, int s) { return griewank_t(n + 1, static_cast<int64_t>(s) + 1) - n; }

struct Builder {
  RevolveSchedule& out;
  std::vector<int> free_slots;

  int take() { const int b = free_slots.back(); free_slots.pop_back(); return b; }
  void give(int b) { free_slots.push_back(b); }

  // every S_t of [i + 1, i + n) recomputed from S_i (slot a) into scratch, reversed at once
  void naive(int i, int n, int a) {
    for (int t = i + n - 1; t > i; --t) {
      out.acts.push_back({RevolveAct::ADV, i, t, a, out.scratch(0)});
      out.acts.push_back({RevolveAct::REV, t, 0, out.scratch(0), 0});
    }
    out.acts.push_back({RevolveAct::REV, i, 0, a, 0});
  }

  // fewest slots su <= s that reach the optimum of n steps, then the smallest split m
  // (0 when su == 0: the naive schedule)
  template <bool TOP>
  void choose(int n, int s, int& su, int& m) const {
    if (s > n) s = n;                     // more slots than steps never help
    const int64_t v = TOP ? G(n, s) : F(n, s);
    su = s;
    while (su > 0 && (TOP ? G(n, su - 1) : F(n, su - 1)) == v) --su;
    m = 0;
    if (su == 0) return;
    for (int k = 1; k < n; ++k) {
      const int64_t c = TOP ? G(n - k, su - 1) + F(k, su) : k + F(n - k, su - 1) + F(k, su);
      if (c == v) { m = k; return; }
    }
    su = 0;                               // unreachable when the closed forms hold
  }

  void rev_f(int i, int n, int a, int s) {
    if (n == 1) { out.acts.push_back({RevolveAct::REV, i, 0, a, 0}); return; }
    int su, m;
    choose<false>(n, s, su, m);
    if (su == 0 || m == 0) { naive(i, n, a); return; }
    const int b = take();
    out.acts.push_back({RevolveAct::ADV, i, i + m, a, b});
    rev_f(i + m, n - m, b, su - 1);
    give(b);
    rev_f(i, m, a, su);
  }

  void rev_g(int i, int n, int a, int s) {
    if (n == 1) { out.acts.push_back({RevolveAct::REV, i, 0, a, 0}); return; }
    int su, m;
    choose<true>(n, s, su, m);
    if (su == 0 || m == 0) { naive(i, n, a); return; }
    const int b = take();
    out.keep[i + m] = b;              // the rollout leaves S_{i+m} in slot b
    rev_g(i + m, n - m, b, su - 1);
    give(b);
    rev_f(i, m, a, su);
  }
};

}  // namespace revolve_detail

// The schedule for T steps and s snapshot slots besides S_0 (s >= 1, T >= 1).
inline RevolveSchedule revolve_schedule(int T, int s) {
  RevolveSchedule r;
  r.T = T;
  r.s = s;
  r.keep.assign(T + 1, -1);
  r.keep[0] = 0;
  revolve_detail::Builder b{r, {}};
  for (int j = s; j >= 1; --j) b.free_slots.push_back(j);
  b.rev_g(0, T, 0, s);
  r.recompute = revolve_detail::G(T, s);
  r.slot_T = r.scratch(0);
  return r;
}

// Forward inner steps the schedule re-runs (for reporting and tests).
inline int64_t revolve_recompute_steps(const RevolveSchedule& r) {
  int64_t n = 0;
  for (const RevolveAct& a : r.acts)
    if (a.kind == RevolveAct::ADV) n += a.t1 - a.t0;
  return n;
}

}  // namespace mf
