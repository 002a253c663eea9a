"""Checkpoint plans of the reverse sweep (mf_checkpoint_plan, host-only: no GPU needed).

The binomial schedule (Section 4's binomial checkpointing) is pinned to Griewank's published
optimum for reversing l steps with c checkpoints, t(l, c) = r l - C(c + r, c + 1) with r the
repetition number, C(c + r - 1, c) < l <= C(c + r, c): in this library's accounting (the
reverse of step t re-runs that step's forward inside the Hessian-vector product, and S_0 is
stored apart from the s snapshot slots) the sweep re-runs t(T + 1, s + 1) - T inner steps."""
from math import comb

import pytest

from paper_2505_00793_gb300 import native


def _griewank(l, c):
    """Minimal forward steps to reverse l steps with c checkpoints (Griewank 1992)."""
    r = 0
    while comb(c + r, c) < l:
        r += 1
    return r * l - comb(c + r, c + 1)


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
