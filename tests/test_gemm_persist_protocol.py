"""Barrier protocol of the persistent CTA-pair GEMM (csrc/tc_gemm_persist.cu), model-checked
on the CPU.

The kernel's three roles are modelled as coroutines over mbarriers with PTX phase semantics
(a barrier completes a phase when its pending arrivals and transaction bytes reach zero;
`try_wait.parity P` succeeds once the phase of parity P has completed).  Asynchronous
completions (TMA bytes, tcgen05.commit arrivals, which keep their issue order) are queued
events.  Random interleavings must finish without deadlock, every MMA must read the stage
data of its own tile and K block, no stage may be refilled before the MMA consumed it, and
no accumulator set may be overwritten before every epilogue warp of both CTAs read it.
The parity and count formulas are the kernel's:
  producer   stage s = g % S, waits empty[s] parity ((g / S) & 1) ^ 1
  MMA        tile j uses set j & 1 (two sets) for the (j >> 1)-th time: waits acc_empty[set]
             parity (use & 1) ^ 1, then full[s] parity (g / S) & 1 per K block
  epilogue   waits acc_full[set] parity use & 1, then arrives on the even CTA's acc_empty[set]
             (count 2 x EPI_WARPS)."""
import random

import numpy as np

import pytest


class Bar:
    def __init__(self, count):
        self.count, self.pending, self.tx, self.k = count, count, 0, 0

    def _check(self):
        if self.pending == 0 and self.tx == 0:
            self.k += 1
            self.pending = self.count

    def arrive(self):
        self.pending -= 1
        assert self.pending >= 0, "more arrivals than the barrier's count"
        self._check()

    def arrive_expect_tx(self, nbytes):
        self.tx += nbytes
        self.arrive()

    def complete_tx(self, nbytes):
        self.tx -= nbytes
        self._check()

    def try_wait(self, parity):
        return (self.k & 1) != parity


class Deadlock(Exception):
    pass


def run_pair(ntiles, pair, npairs, nk, stages, nsets, epi_warps, seed,
             acc_empty_count=None, mma_parity_flip=0):
    """One CTA pair of the persistent kernel; returns the number of tiles it drained."""
    rnd = random.Random(seed)
    full0 = [Bar(1) for _ in range(stages)]                       # even CTA only
    empty = [[Bar(1) for _ in range(stages)] for _ in range(2)]   # both CTAs
    acc_full = [[Bar(1) for _ in range(2)] for _ in range(2)]
    acc_empty0 = [Bar(acc_empty_count or 2 * epi_warps) for _ in range(2)]
    stage_data = [[None] * stages for _ in range(2)]
    consumed, reads, acc = set(), {}, [None, None]
    events = []
    tiles = list(range(pair, ntiles, npairs))

    def set_use(j):
        return (j & 1, j >> 1) if nsets == 2 else (0, j)

    def producer(rank):
        g = 0
        for t in tiles:
            for i in range(nk):
                s, ph = g % stages, (g // stages) & 1
                while not empty[rank][s].try_wait(ph ^ 1):
                    yield
                assert g < stages or (g - stages) in consumed, "stage refilled before consumed"
                if rank == 0:
                    full0[s].arrive_expect_tx(2)
                stage_data[rank][s] = (t, i)
                events.append(("tx", s))
                g += 1
                yield

    def mma():
        for j, t in enumerate(tiles):
            st, use = set_use(j)
            while not acc_empty0[st].try_wait((use & 1) ^ 1 ^ mma_parity_flip):
                yield
            assert use == 0 or reads.get((st, use - 1), 0) == 2 * epi_warps, \
                "accumulator set overwritten before the epilogue read it"
            acc[st] = [t, []]
            for i in range(nk):
                g = j * nk + i
                s, ph = g % stages, (g // stages) & 1
                while not full0[s].try_wait(ph):
                    yield
                assert stage_data[0][s] == (t, i) and stage_data[1][s] == (t, i), "stage data"
                acc[st][1].append(i)
                events.append(("commit_stage", s, g))
                yield
            events.append(("commit_acc", st))
            yield

    def epilogue(rank):
        for j, t in enumerate(tiles):
            st, use = set_use(j)
            while not acc_full[rank][st].try_wait(use & 1):
                yield
            assert acc[st] == [t, list(range(nk))], "epilogue read an unfinished tile"
            yield
            reads[(st, use)] = reads.get((st, use), 0) + 1
            acc_empty0[st].arrive()
            yield

    actors = [producer(0), producer(1), mma()]
    actors += [epilogue(r) for r in (0, 1) for _ in range(epi_warps)]
    steps = 0
    while actors or events:
        c = rnd.randrange(len(actors) + (1 if events else 0))
        if c == len(actors):
            commits = [k for k, e in enumerate(events) if e[0] != "tx"]
            tx = [k for k, e in enumerate(events) if e[0] == "tx"]
            # TMA bytes land in any order; tcgen05.commit arrivals keep their issue order
            idx = commits[0] if commits and (not tx or rnd.random() < 0.5) else rnd.choice(tx)
            ev = events.pop(idx)
            if ev[0] == "tx":
                full0[ev[1]].complete_tx(1)
            elif ev[0] == "commit_stage":
                consumed.add(ev[2])
                empty[0][ev[1]].arrive()
                empty[1][ev[1]].arrive()
            else:
                acc_full[0][ev[1]].arrive()
                acc_full[1][ev[1]].arrive()
            continue
        try:
            next(actors[c])
        except StopIteration:
            actors.pop(c)
        steps += 1
        if steps > 200000:
            raise Deadlock()
    # tiles whose accumulators every epilogue warp of both CTAs read
    return sum(1 for n in reads.values() if n == 2 * epi_warps)


def _configs(n):
    rnd = random.Random(12345)
    for seed in range(n):
        npairs = rnd.randint(1, 4)
        yield dict(ntiles=rnd.randint(1, 12), pair=rnd.randrange(npairs), npairs=npairs,
                   nk=rnd.randint(1, 7), stages=rnd.randint(2, 6), nsets=rnd.choice([1, 2]),
                   epi_warps=rnd.choice([1, 2, 8, 12]), seed=seed)


def test_protocol_completes_every_tile():
    for cfg in _configs(400):
        expect = len(range(cfg["pair"], cfg["ntiles"], cfg["npairs"]))
        assert run_pair(**cfg) == expect, cfg


@pytest.mark.parametrize("mistake", ["acc_empty_count", "mma_parity"])
def test_model_catches_planted_mistakes(mistake):
    """A wrong arrival count or a flipped parity on the accumulator hand-off is caught in
    (nearly) every configuration where a set is reused."""
    caught = eligible = 0
    for cfg in _configs(60):
        if len(range(cfg["pair"], cfg["ntiles"], cfg["npairs"])) < 3:
            continue
        eligible += 1
        kw = dict(cfg)
        if mistake == "acc_empty_count":
            kw["acc_empty_count"] = cfg["epi_warps"] + 1 if cfg["epi_warps"] > 1 else 3
        else:
            kw["mma_parity_flip"] = 1
        try:
            run_pair(**kw)
        except (AssertionError, Deadlock):
            caught += 1
    assert eligible > 20 and caught >= 0.9 * eligible, (caught, eligible)


# ---- index arithmetic of the persistent kernel ---------------------------------------------
BM, BK = 128, 64


def _persist_coverage(M, N, BN, batch, npairs, epi_warps=12):
    """Every output element written by the kernel's epilogue mapping, and the TMA boxes each
    CTA loads, for one launch (the kernel's formulas restated).  epi_warps epilogue warps
    (8 for the backward epilogues, 12 otherwise): epi_warps / 4 per TMEM lane quadrant,
    taking the quadrant's 16-column chunks in turn."""
    tiles_n = -(-N // BN)
    pairs_m = -(-M // (2 * BM))
    ntiles = tiles_n * pairs_m * batch
    BH = BN // 2
    written = np.zeros((batch, M, N), np.int32)
    a_rows, b_rows = set(), set()
    groups = epi_warps // 4
    for pair in range(npairs):
        for t in range(pair, ntiles, npairs):
            # grouped order of the kernel: groups of up to 8 row blocks, rows fastest
            group = min(pairs_m, 8)
            bz, r = divmod(t, tiles_n * pairs_m)
            g, w = divmod(r, group * tiles_n)
            rows = min(group, pairs_m - g * group)
            mp, tn = g * group + w % rows, w // rows
            for rank in (0, 1):
                m0 = mp * 2 * BM + rank * BM
                a_rows.add((bz, m0))
                b_rows.add((bz, tn * BN + rank * BH))
                n0 = tn * BN
                for warp in range(2, 2 + epi_warps):
                    q = warp & 3
                    c_begin = ((warp - 2) >> 2) * 16
                    for lane in range(32):
                        row = m0 + q * 32 + lane
                        for c in range(c_begin, BN, 16 * groups):
                            if n0 + c >= N or row >= M:
                                continue
                            cols = [n0 + c + j for j in range(16) if n0 + c + j < N]
                            written[bz, row, cols] += 1
    return written, a_rows, b_rows, pairs_m, tiles_n


@pytest.mark.parametrize("epi_warps", [8, 12])
@pytest.mark.parametrize("M,N,BN,batch,npairs", [
    (256, 128, 128, 1, 1), (300, 520, 128, 1, 3), (1000, 130, 256, 1, 76),
    (1025, 1024, 256, 1, 7), (600, 1000, 128, 3, 5), (2048, 1024, 128, 1, 76),
    (2900, 520, 128, 2, 9)])
def test_persistent_tiles_cover_every_output_once(M, N, BN, batch, npairs, epi_warps):
    written, a_rows, b_rows, pairs_m, tiles_n = _persist_coverage(M, N, BN, batch, npairs,
                                                                  epi_warps)
    assert (written == 1).all()
    # A boxes: 128 rows per CTA from every 256-row block; B boxes: BN/2 rows per CTA
    assert {m for _, m in a_rows} == {mp * 2 * BM + r * BM for mp in range(pairs_m) for r in (0, 1)}
    assert {n for _, n in b_rows} == {tn * BN + r * BN // 2 for tn in range(tiles_n) for r in (0, 1)}
    # TMA x coordinates: K offsets i * 64 (bf16: 128-byte multiples); MN-major boxes start at
    # row offsets that are multiples of 64 elements
    assert all(m % 64 == 0 for _, m in a_rows) and all(n % 64 == 0 for _, n in b_rows)


def test_persistent_tmem_columns_fit():
    """Accumulator sets and blocks as the launcher sizes them stay inside the 512 TMEM
    columns it allocates, for every tile width and product count the kernel takes."""
    def acc_blocks(nlogical, bn):
        return 4 if nlogical * 4 * bn <= 512 else 2 if nlogical * 2 * bn <= 512 else 1

    def persist_nsub(nacc, bn):
        for n in (4, 2, 1):
            if 2 * nacc * n * bn <= 512:
                return n
        return acc_blocks(nacc, bn)

    for bn in (128, 256):
        for nacc in (1, 2):
            nsub = persist_nsub(nacc, bn)
            nsets = 2 if 2 * nacc * nsub * bn <= 512 else 1
            set_cols = nacc * nsub * bn
            assert nsets * set_cols <= 512
            # highest column an MMA writes: set (nsets-1), block nacc*nsub-1, BN columns
            assert (nsets - 1) * set_cols + (nacc * nsub - 1) * bn + bn <= 512
            assert nsub & (nsub - 1) == 0   # the rotation masks with nsub - 1
