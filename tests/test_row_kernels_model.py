"""Index arithmetic and summation order of the decoder's token-ordering and embedding-gradient
kernels (csrc/decoder_kernels.cu), restated on the CPU.

- scan_kernel: thread t of 1024 owns counts [t per, (t + 1) per); run totals are scanned
  within warps by shuffles, then over the 32 warp totals; the thread writes its run's
  exclusive starts, and start[V] is the total.  Must equal the exclusive prefix sum.
- token_order_kernel: ids are dealt to G blocks with a stride; each id's scattered positions
  (any order) are ranked: segments of up to 32 by counting smaller positions in a warp,
  longer ones through a bitmap of positions (rank = set bits below the position, with the
  words' bit counts prefix-summed by 256 threads) when the batch has at most 65536 tokens.
  Must equal a stable sort of the token ids.
- rmsnorm_bwd_warp_kernel + gain_grad_final_kernel: every (row, column) of the gain gradient is
  added into exactly one partial row, and every partial row read once by the final sums.
- embed_bwd_kernel: a segment of up to 8 rows is summed by one warp in row order from zero; a
  longer one by eight warps over contiguous parts, the parts added in warp order.  For up to
  8 rows both give the same float32 bits."""
import numpy as np
import pytest

from paper_2505_00793_gb300 import synth

SCAN_THREADS = 1024


def scan_model(count):
    V = len(count)
    per = -(-V // SCAN_THREADS)
    runs = [int(np.sum(count[t * per:min(V, t * per + per)], dtype=np.int64))
            for t in range(SCAN_THREADS)]
    inc = []
    for w in range(SCAN_THREADS // 32):
        acc = 0
        for lane in range(32):
            acc += runs[w * 32 + lane]
            inc.append(acc)
    wtot = np.cumsum([inc[w * 32 + 31] for w in range(SCAN_THREADS // 32)]).tolist()
    start = [0] * (V + 1)
    for t in range(SCAN_THREADS):
        w = t // 32
        acc = inc[t] - runs[t] + (wtot[w - 1] if w > 0 else 0)
        for i in range(t * per, min(V, t * per + per)):
            start[i] = acc
            acc += int(count[i])
    start[V] = wtot[-1]
    return start


def order_model(V, N, start, tmp, G, bitmap_tokens=32 * 2048):
    order = [None] * N
    use_bm = N <= bitmap_tokens
    nw = (N + 31) >> 5
    per = (nw + 255) // 256
    for b in range(G):
        nmine = (V - b + G - 1) // G
        for k0 in range(0, nmine, 256):
            for t in range(min(256, nmine - k0)):
                v = b + (k0 + t) * G
                a, L = start[v], start[v + 1] - start[v]
                if L == 0:
                    continue
                seg = tmp[a:a + L]
                if L <= 32 or not use_bm:
                    for p in seg:
                        order[a + sum(1 for q in seg if q < p)] = p
                    continue
                bm = [0] * nw
                for p in seg:
                    bm[p >> 5] |= 1 << (p & 31)
                wpre, acc = [0] * nw, 0
                for th in range(256):
                    for j in range(th * per, min(nw, th * per + per)):
                        wpre[j] = acc
                        acc += bin(bm[j]).count("1")
                for p in seg:
                    wd = p >> 5
                    order[a + wpre[wd] + bin(bm[wd] & ((1 << (p & 31)) - 1)).count("1")] = p
    return order


@pytest.mark.parametrize("V", [1, 2, 7, 1024, 1025, 32768, 40000])
def test_scan_is_exclusive_prefix_sum(V):
    rng = np.random.default_rng(V)
    count = rng.integers(0, 9, V)
    ref = np.concatenate([[0], np.cumsum(count)]).tolist()
    assert scan_model(count) == ref


@pytest.mark.parametrize("V,N,bitmap", [(32768, 8192, True), (256, 600, True), (2, 50, True),
                                        (1000, 4096, True), (1000, 4096, False)])
def test_ordering_is_stable_sort(V, N, bitmap):
    """Zipf(1.1) ids as the workloads draw them; the scatter fills each segment in a random
    order (atomic slots), as the GPU may.  bitmap=False takes the counting path of batches
    above 65536 tokens on a small batch."""
    rng = np.random.default_rng(N)
    ids = synth.zipf_ids(rng, (N,), V, 1.1)
    count = np.bincount(ids, minlength=V)
    start = scan_model(count)
    tmp, slots = [None] * N, count.copy()
    for r in rng.permutation(N):
        i = ids[r]
        slots[i] -= 1
        tmp[start[i] + slots[i]] = int(r)
    order = order_model(V, N, start, tmp, min(V, 304), 32 * 2048 if bitmap else 0)
    assert order == np.argsort(ids, kind="stable").tolist()
    if N == 8192:
        assert count.max() > 32   # the bitmap path runs (the most frequent id's segment)


def _block_sum(rows):
    cnt = len(rows)
    parts = []
    for w in range(8):
        acc = np.zeros(4, np.float32)
        for r in range((w * cnt) // 8, ((w + 1) * cnt) // 8):
            acc = (acc + rows[r]).astype(np.float32)
        parts.append(acc)
    t = parts[0]
    for p in parts[1:]:
        t = (t + p).astype(np.float32)
    return t


def _warp_sum(rows):
    acc = np.zeros(4, np.float32)
    for r in rows:
        acc = (acc + r).astype(np.float32)
    return acc


def test_short_segment_sum_matches_block_partition_bitwise():
    rng = np.random.default_rng(0)
    specials = np.array([0.0, -0.0, 1e-38, -1e-38, 3.0e38, -3.0e38], np.float32)
    for trial in range(3000):
        cnt = int(rng.integers(1, 9))
        rows = rng.standard_normal((cnt, 4)).astype(np.float32) * np.float32(10.0) ** \
            rng.integers(-3, 4, (cnt, 4)).astype(np.float32)
        if trial % 3 == 0:
            mask = rng.random((cnt, 4)) < 0.3
            rows[mask] = rng.choice(specials, mask.sum())
        with np.errstate(over="ignore"):
            b, w = _block_sum(rows), _warp_sum(rows)
        assert b.tobytes() == w.tobytes(), (cnt, rows, b, w)


@pytest.mark.parametrize("N,d", [(2048, 1024), (13, 64), (64, 1000), (9, 8), (250, 4096)])
def test_gain_partials_cover_every_row_and_column_once(N, d):
    """The RMSNorm backward's gain pass: block b (eight rows), warp w, lane l takes columns
    w*128 + 4l + 1024k .. + 3 and adds rows 8b .. min(N, 8b + 8) into partial row b; the final
    kernel's thread (x, y) of block g reads partial rows y, y + 32, ... of column 32g + x."""
    nblk = (N + 7) // 8
    contrib = np.zeros((N, d), np.int32)
    written = np.zeros((nblk, d), np.int32)
    for b in range(nblk):
        q0, q1 = 8 * b, min(N, 8 * b + 8)
        for w in range(8):
            for lane in range(32):
                for c in range(w * 128 + lane * 4, d, 1024):
                    written[b, c:c + 4] += 1
                    contrib[q0:q1, c:c + 4] += 1
    assert (written == 1).all() and (contrib == 1).all()
    read = np.zeros((nblk, d), np.int32)
    for g in range((d + 31) // 32):
        for x in range(32):
            j = g * 32 + x
            if j >= d:
                continue
            for y in range(32):
                for c in range(y, nblk, 32):
                    read[c, j] += 1
    assert (read == 1).all()
