"""Checkpoint plans of the reverse sweep (mf_checkpoint_plan, host-only: no GPU needed).

The binomial schedule (Section 4's binomial checkpointing) is pinned to Griewank's published
optimum for reversing l steps with c checkpoints, t(l, c) = r l - C(c + r, c + 1) with r the
repetition number, C(c + r - 1, c) < l <= C(c + r, c): in this library's accounting (the
reverse of step t re-runs that step's forward inside the Hessian-vector product, and S_0 is
stored apart from the s snapshot slots) the sweep re-runs t(T + 1, s + 1) - T inner steps."""
import os
import shutil
import subprocess
from functools import lru_cache
from math import comb

import pytest

from paper_2505_00793_gb300 import native


def _griewank(l, c):
    """Minimal forward steps to reverse l steps with c checkpoints (Griewank 1992)."""
    r = 0
    while comb(c + r, c) < l:
        r += 1
    return r * l - comb(c + r, c + 1)


@lru_cache(maxsize=None)
def _recursion(n, s, top):
    """The split-point recursion itself, by brute force: F (top=False) reverses n steps
    from a stored S_i with s free slots, each split paying m steps to advance; G (top=True)
    splits the rolled-out top level, whose advances are free."""
    if n == 1:
        return 0
    if s == 0:
        return n * (n - 1) // 2
    best = _recursion(n, s - 1, top)
    for m in range(1, n):
        c = _recursion(n - m, s - 1, top) + _recursion(m, s, False) + (0 if top else m)
        best = min(best, c)
    return best


def _plan(T, k=1, s=0):
    try:
        return native.checkpoint_plan(T, k, s)
    except ImportError:
        pytest.skip("native library not built")


@pytest.mark.parametrize("T", [1, 2, 3, 7, 16, 32, 100])
def test_binomial_recompute_is_griewank_optimum(T):
    for s in range(1, 12):
        slots, re = _plan(T, 1, s)
        assert re == _griewank(T + 1, min(s, max(T - 1, 1)) + 1) - T, (T, s, re)
        assert slots == min(s, max(T - 1, 1)) + 3


def test_binomial_recompute_is_recursion_optimum():
    # the library builds its schedule from closed forms; the recursion they solve, by brute force
    for T in range(1, 41):
        for s in range(1, 9):
            sb = min(s, max(T - 1, 1))
            assert _plan(T, 1, s)[1] == _recursion(T, sb, True), (T, s)


def test_binomial_schedule_replays():
    """Replays the library's schedules slot by slot on the host (tests/revolve_check.cpp)."""
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not found")
    here = os.path.dirname(os.path.abspath(__file__))
    csrc = os.path.join(os.path.dirname(here), "paper_2505_00793_gb300", "csrc")
    exe = os.path.join(os.environ.get("TMPDIR", "/tmp"), f"revolve_check_{os.getpid()}")
    subprocess.run([gxx, "-std=c++17", "-O2", "-I", csrc, os.path.join(here, "revolve_check.cpp"),
                    "-o", exe], check=True)
    try:
        out = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    finally:
        if os.path.exists(exe):
            os.remove(exe)
    assert out.returncode == 0 and "bad=0" in out.stdout, out.stdout[-2000:]


def test_binomial_plan_is_fast_at_the_limits():
    # the closed forms keep the largest schedule (T = 4096, s = 1024) to milliseconds
    import time
    t0 = time.perf_counter()
    slots, re = _plan(4096, 1, 1024)
    assert time.perf_counter() - t0 < 5.0
    assert (slots, re) == (1027, _griewank(4097, 1025) - 4096)


def test_binomial_trade_off():
    # more slots never cost more recomputation; T - 1 snapshots recompute nothing
    for T in (5, 16, 33):
        re = [_plan(T, 1, s)[1] for s in range(1, T + 2)]
        assert all(a >= b for a, b in zip(re, re[1:]))
        assert re[T - 2] == 0
    # the deep workload's T = 32: uniform segments of 6 keep 11 states and re-run 25 steps;
    # the binomial schedule re-runs as few with 9 states, and fewer (23) with the same 11
    assert _plan(32, 6, 0) == (11, 25)
    assert _plan(32, 1, 6) == (9, 25)
    assert _plan(32, 1, 8) == (11, 23)


def test_uniform_and_full_plans():
    assert _plan(32, 1, 0) == (33, 0)
    assert _plan(32, 0, 0) == (33, 0)
    assert _plan(16, 4, 0) == (4 + 4, 3 * 3)
    assert _plan(7, 3, 0) == (2 + 3, 2 * 2)
    assert _plan(5, 9, 0) == (1 + 5, 0)      # k > T acts as T


@pytest.mark.parametrize("args", [(0, 1, 0), (8, -1, 0), (8, 1, -1), (8, 2, 3),
                                  (5000, 1, 2), (8, 1, 2000)])
def test_invalid_plans_are_rejected(args):
    try:
        native.lib()
    except ImportError:
        pytest.skip("native library not built")
    with pytest.raises(native.MixflowError):
        native.checkpoint_plan(*args)
