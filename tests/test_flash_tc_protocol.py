"""Barrier protocols of the tcgen05 fused attention (csrc/flash_tc.cu), model-checked on the CPU.

Each role of a CTA is a coroutine over mbarriers with PTX phase semantics (the `Bar` model of
tests/test_gemm_persist_protocol.py: a phase completes when its pending arrivals and
transaction bytes reach zero; `try_wait.parity P` succeeds once the phase of parity P has
completed).  TMA bytes land in any order; tcgen05.commit arrivals keep their issue order.  An
MMA is taken to write its TMEM accumulator or read its shared-memory operands at any time
between its issue and its commit, so the checks are:
- nobody reads a TMEM score tile, a stage or an A-operand tile that a later write has been
  issued over, or before the write it needs has committed;
- no stage is refilled, and no A-operand tile rewritten, while an issued MMA may still read it;
- random interleavings end without deadlock, and the outputs are read after the last
  accumulating product committed.

Backward (key-tile and query-tile kernels, one protocol):
  producer   resident tiles once (res_full); query tile i into stage i % 2: waits
             st_empty[s] parity ((i / 2) & 1) ^ 1
  MMA        res_full parity 0; scores(0); per tile i: s_free parity i & 1, then scores(i + 1)
             (st_full parity ((i + 1) / 2) & 1, commit s_full), p_full parity i & 1, the
             accumulating products (commit st_empty[i % 2], then o_done)
  8 warps    s_full parity i & 1; read the scores; arrive s_free; read the stage's row
             statistics; for i > 0 o_done parity (i - 1) & 1; write the A operands; arrive
             p_full; at the end o_done parity (n - 1) & 1, then the outputs
Forward (one or two stages):
  MMA        q_full; per key tile j: kv_full, for j > 0 s_free parity (j - 1) & 1, S (commit
             s_full), p_full parity j & 1, the P V products (commit kv_empty, then o_done)
  4 warps    s_full parity j & 1; read S; for j > 0 o_done parity (j - 1) & 1 (rescale O);
             write P; arrive s_free and p_full; at the end o_done parity (n - 1) & 1."""
import random

import pytest

from test_gemm_persist_protocol import Bar, Deadlock


def _schedule(actors, events, on_event, rnd, limit=20000):
    steps = 0
    while actors or events:
        c = rnd.randrange(len(actors) + (1 if events else 0))
        if c == len(actors):
            commits = [k for k, e in enumerate(events) if e[0] != "tx"]
            tx = [k for k, e in enumerate(events) if e[0] == "tx"]
            idx = commits[0] if commits and (not tx or rnd.random() < 0.5) else rnd.choice(tx)
            on_event(events.pop(idx))
            continue
        try:
            next(actors[c])
        except StopIteration:
            actors.pop(c)
        steps += 1
        if steps > limit:
            raise Deadlock()


def run_backward(ntile, seed, ew=8, stages=2, s_free_count=None, ew_o_done_flip=0,
                 early_scores=False):
    """One CTA of the tcgen05 attention backward over ntile streamed tiles."""
    rnd = random.Random(seed)
    res_full = Bar(1)
    st_full = [Bar(1) for _ in range(stages)]
    st_empty = [Bar(1) for _ in range(stages)]
    s_full, o_done = Bar(1), Bar(1)
    s_free, p_full = Bar(s_free_count or ew), Bar(ew)
    st = {"stage": [None] * stages, "stage_readers": [set() for _ in range(stages)],
          "S_issued": None, "S_done": None, "op": [None] * ew, "op_reading": None,
          "acc_done": -1, "outputs": 0}
    events = []

    def producer():
        events.append(("tx", "res"))
        res_full.arrive_expect_tx(1)
        yield
        for i in range(ntile):
            s, ph = i % stages, (i // stages) & 1
            while not st_empty[s].try_wait(ph ^ 1):
                yield
            assert not st["stage_readers"][s], "stage refilled while an MMA may read it"
            st_full[s].arrive_expect_tx(1)
            st["stage"][s] = i
            events.append(("tx", s))
            yield

    def scores(i):
        s = i % stages
        while not st_full[s].try_wait((i // stages) & 1):
            yield
        assert st["stage"][s] == i, "scores read the wrong stage"
        st["S_issued"] = i
        st["stage_readers"][s].add(("S", i))
        events.append(("commit", "s_full", i))
        yield

    def mma():
        while not res_full.try_wait(0):
            yield
        yield from scores(0)
        for i in range(ntile):
            if early_scores and i + 1 < ntile:
                yield from scores(i + 1)
            while not s_free.try_wait(i & 1):
                yield
            if not early_scores and i + 1 < ntile:
                yield from scores(i + 1)
            while not p_full.try_wait(i & 1):
                yield
            assert all(o == i for o in st["op"]), "products read A operands of another tile"
            s = i % stages
            assert st["stage"][s] == i, "products read the wrong stage"
            st["stage_readers"][s].add(("acc", i))
            st["op_reading"] = i
            events.append(("commit", "st_empty", i))
            events.append(("commit", "o_done", i))
            yield

    def ew_warp(w):
        for i in range(ntile):
            while not s_full.try_wait(i & 1):
                yield
            assert st["S_done"] == i and st["S_issued"] == i, "scores read before written"
            yield
            assert st["S_issued"] == i, "scores overwritten while being read"
            s_free.arrive()
            assert st["stage"][i % stages] == i, "row statistics read from a refilled stage"
            yield
            if i > 0:
                while not o_done.try_wait(((i - 1) & 1) ^ ew_o_done_flip):
                    yield
            assert st["op_reading"] is None, "A operands rewritten while the products read them"
            st["op"][w] = i
            p_full.arrive()
            yield
        while not o_done.try_wait((ntile - 1) & 1):
            yield
        assert st["acc_done"] == ntile - 1, "outputs read before the last products"
        st["outputs"] += 1

    def on_event(ev):
        if ev[0] == "tx":
            (res_full if ev[1] == "res" else st_full[ev[1]]).complete_tx(1)
        elif ev[1] == "s_full":
            st["S_done"] = ev[2]
            st["stage_readers"][ev[2] % stages].discard(("S", ev[2]))
            s_full.arrive()
        elif ev[1] == "st_empty":
            st["stage_readers"][ev[2] % stages].discard(("acc", ev[2]))
            st_empty[ev[2] % stages].arrive()
        else:
            st["op_reading"] = None
            st["acc_done"] = ev[2]
            o_done.arrive()

    _schedule([producer(), mma()] + [ew_warp(w) for w in range(ew)], events, on_event, rnd)
    return st["outputs"]


def run_forward(nkt, seed, stages=1, warps=4, o_done_flip=0, s_free_late=True,
                p_full_count=None):
    """One CTA of the tcgen05 attention forward over nkt key tiles."""
    rnd = random.Random(seed)
    q_full = Bar(1)
    kv_full = [Bar(1) for _ in range(stages)]
    kv_empty = [Bar(1) for _ in range(stages)]
    s_full, o_done = Bar(1), Bar(1)
    s_free, p_full = Bar(warps), Bar(p_full_count or warps)
    st = {"stage": [None] * stages, "stage_readers": [set() for _ in range(stages)],
          "S_issued": None, "S_done": None, "P": [None] * warps, "P_reading": None,
          "O_writer": None, "O_done": -1, "outputs": 0}
    events = []

    def producer():
        q_full.arrive_expect_tx(1)
        events.append(("tx", "q"))
        yield
        for j in range(nkt):
            s, ph = j % stages, (j // stages) & 1
            while not kv_empty[s].try_wait(ph ^ 1):
                yield
            assert not st["stage_readers"][s], "K/V stage refilled while an MMA may read it"
            kv_full[s].arrive_expect_tx(1)
            st["stage"][s] = j
            events.append(("tx", s))
            yield

    def mma():
        while not q_full.try_wait(0):
            yield
        for j in range(nkt):
            s = j % stages
            while not kv_full[s].try_wait((j // stages) & 1):
                yield
            if j > 0 and s_free_late:
                while not s_free.try_wait((j - 1) & 1):
                    yield
            assert st["stage"][s] == j
            st["S_issued"] = j
            st["stage_readers"][s].add(("S", j))
            events.append(("commit", "s_full", j))
            yield
            while not p_full.try_wait(j & 1):
                yield
            assert all(p == j for p in st["P"]), "P V read P of another tile"
            st["stage_readers"][s].add(("PV", j))
            st["P_reading"] = j
            st["O_writer"] = j
            events.append(("commit", "kv_empty", j))
            events.append(("commit", "o_done", j))
            yield

    def softmax(w):
        for j in range(nkt):
            while not s_full.try_wait(j & 1):
                yield
            assert st["S_done"] == j and st["S_issued"] == j, "S read before written"
            yield
            assert st["S_issued"] == j, "S overwritten while being read"
            if j > 0:
                while not o_done.try_wait(((j - 1) & 1) ^ o_done_flip):
                    yield
                # rescaling O in TMEM: no P V product may be writing it
                assert st["O_writer"] is None, "O rescaled while a product writes it"
            assert st["P_reading"] is None, "P rewritten while P V reads it"
            st["P"][w] = j
            yield
            s_free.arrive()
            p_full.arrive()
            yield
        while not o_done.try_wait((nkt - 1) & 1):
            yield
        assert st["O_done"] == nkt - 1, "outputs read before the last P V product"
        st["outputs"] += 1

    def on_event(ev):
        if ev[0] == "tx":
            (q_full if ev[1] == "q" else kv_full[ev[1]]).complete_tx(1)
        elif ev[1] == "s_full":
            st["S_done"] = ev[2]
            st["stage_readers"][ev[2] % stages].discard(("S", ev[2]))
            s_full.arrive()
        elif ev[1] == "kv_empty":
            st["stage_readers"][ev[2] % stages].discard(("PV", ev[2]))
            kv_empty[ev[2] % stages].arrive()
        else:
            st["P_reading"] = None
            st["O_writer"] = None
            st["O_done"] = ev[2]
            o_done.arrive()

    _schedule([producer(), mma()] + [softmax(w) for w in range(warps)], events, on_event, rnd)
    return st["outputs"]


def test_backward_protocol_completes():
    rnd = random.Random(7)
    for seed in range(300):
        n = rnd.randint(1, 9)
        assert run_backward(n, seed) == 8, (n, seed)


@pytest.mark.parametrize("stages", [1, 2])
def test_forward_protocol_completes(stages):
    rnd = random.Random(11)
    for seed in range(300):
        n = rnd.randint(1, 9)
        assert run_forward(n, seed, stages=stages) == 4, (n, seed)


@pytest.mark.parametrize("mistake", ["s_free_count", "o_done_parity", "early_scores"])
def test_backward_model_catches_planted_mistakes(mistake):
    """A wrong arrival count, a flipped parity or the next tile's scores issued before the
    warps have read this tile's are caught in nearly every run with several tiles."""
    caught = runs = 0
    rnd = random.Random(3)
    for seed in range(80):
        n = rnd.randint(3, 9)
        kw = {"s_free_count": 9} if mistake == "s_free_count" else \
             {"ew_o_done_flip": 1} if mistake == "o_done_parity" else {"early_scores": True}
        runs += 1
        try:
            run_backward(n, seed, **kw)
        except (AssertionError, Deadlock):
            caught += 1
    assert caught >= 0.9 * runs, (mistake, caught, runs)


@pytest.mark.parametrize("mistake", ["o_done_parity", "p_full_count"])
def test_forward_model_catches_planted_mistakes(mistake):
    caught = runs = 0
    rnd = random.Random(5)
    for seed in range(80):
        n = rnd.randint(3, 9)
        kw = {"o_done_flip": 1} if mistake == "o_done_parity" else {"p_full_count": 5}
        runs += 1
        try:
            run_forward(n, seed, stages=2, **kw)
        except (AssertionError, Deadlock):
            caught += 1
    assert caught >= 0.9 * runs, (mistake, caught, runs)


def test_forward_s_free_wait_is_implied_by_p_full():
    """The forward MMA thread's wait on s_free before the next tile's scores never holds it
    back: the softmax warps arrive on s_free and p_full together, and the MMA thread has
    already waited on p_full of the previous tile before it issued that tile's P V products.
    Without the wait the protocol stays correct."""
    rnd = random.Random(13)
    for seed in range(200):
        n = rnd.randint(1, 9)
        assert run_forward(n, seed, stages=rnd.choice([1, 2]), s_free_late=False) == 4
