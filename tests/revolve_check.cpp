// Replays binomial checkpoint schedules on the host and checks them: every advance starts
// from the state its source slot holds and never writes the slot it reads, every reverse
// finds S_t in its slot, the reverses run t = T-1, ..., 0 in order, and the steps re-run
// add up to the schedule's own count.  Prints "bad=<n>" and exits non-zero on a failure.
// Built and run by tests/test_checkpoint_plan.py.
#include <revolve.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <vector>

static int check(int T, int s) {
  const mf::RevolveSchedule r = mf::revolve_schedule(T, s);
  int bad = 0;
  std::vector<int> held(r.n_slots(), -1);   // the t of the S_t each slot holds
  held[0] = 0;
  // an advance ping-pongs through the scratch slots and ends in its destination
  auto advance = [&](int t0, int t1, int src, int dst) {
    if (held[src] != t0) ++bad;
    const int other = dst == r.scratch(0) ? r.scratch(1) : r.scratch(0);
    int cur = src;
    for (int k = 0, n = t1 - t0; k < n; ++k) {
      const int out = (n - 1 - k) % 2 == 0 ? dst : other;
      if (out == cur) ++bad;
      held[out] = t0 + k + 1;
      cur = out;
    }
  };
  int at = 0, cur = 0;
  for (int t = 1; t < T; ++t)
    if (r.keep[t] >= 0) { advance(at, t, cur, r.keep[t]); at = t; cur = r.keep[t]; }
  advance(at, T, cur, r.slot_T);
  if (held[r.slot_T] != T) ++bad;
  long long re = 0;
  int next = T - 1;
  for (const mf::RevolveAct& a : r.acts) {
    if (a.kind == mf::RevolveAct::ADV) {
      if (a.src > r.s) ++bad;                 // advances start from a kept state
      advance(a.t0, a.t1, a.src, a.dst);
      re += a.t1 - a.t0;
    } else {
      if (a.t0 != next || held[a.src] != a.t0) ++bad;
      --next;
    }
  }
  if (next != -1 || re != r.recompute) ++bad;
  if (bad) std::printf("T=%d s=%d: %d errors\n", T, s, bad);
  return bad;
}

int main() {
  int bad = 0;
  for (int T = 1; T <= 64; ++T)
    for (int s = 1; s <= 16; ++s) bad += check(T, std::min(s, std::max(T - 1, 1)));
  const int large[][2] = {{4096, 1}, {4096, 3}, {4096, 64}, {4096, 1024}, {1000, 7}};
  for (const auto& c : large) bad += check(c[0], c[1]);
  std::printf("bad=%d\n", bad);
  return bad ? EXIT_FAILURE : EXIT_SUCCESS;
}
