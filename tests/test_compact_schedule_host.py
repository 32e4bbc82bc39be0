"""The in-place compaction (the index-gather of Sec. 5.3) on the CPU: the facts its ordering
rests on, and the pieces of compact_kernel that decide where it reads and writes.

compact_kernel moves slot j <- row kept[j] tile by tile: a tile's rows are gathered with
asynchronous copies into a ring of shared-memory stages (several tiles ahead) and written back
by one bulk copy once all of the tile's copies have landed.  It needs no other ordering
because (a) kept is strictly increasing with kept[j] >= j, so every row a slot of tile i is
read for belongs to a tile <= i, and (b) every row read for a later tile lies above every slot
of tile i.  Both are checked on the oracle's retained sets and on random lists; the kernel's
32-way search for the first moved slot is restated and checked against a linear scan; and the
kernel's source is checked to keep its waits, fence, barrier and store in that order.
"""
import os
import re

import numpy as np

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def first_moved(kept):
    j = 0
    while j < len(kept) and kept[j] == j:
        j += 1
    return j


def search32(kept, cnt):
    """the kernel's 32-way search: probes lo + lane * step of every lane, ballot, narrow"""
    lo, hi = 0, cnt
    rounds = 0
    while lo < hi:
        rounds += 1
        step = (hi - lo + 31) >> 5
        hits = [lo + lane * step < hi and kept[lo + lane * step] != lo + lane * step
                for lane in range(32)]
        if any(hits):
            f = hits.index(True)
            hi = lo + f * step
            if f:
                lo += (f - 1) * step + 1
        else:
            lo += min(31, (hi - 1 - lo) // step) * step + 1
    return lo, rounds


def keep_cases():
    prm = oracle.params()
    rng = np.random.default_rng(7)
    cases = [(8193, 4096, 0, (0, 0), 0), (131073, 32768, 0, (0, 0), 0),
             (131073, 32768, 1, (114689, 131073), 0), (32769, 8192, 1, (32000, 32600), 1),
             (5000, 4096, 1, (4900, 4940), 0), (5000, 4096, 1, (4800, 4864), 0),
             (4097, 4096, 0, (0, 0), 0), (300, 256, 0, (0, 0), 0)]
    for _ in range(60):
        B = int(rng.choice([256, 1024, 4096, 8192]))
        n = int(rng.integers(B + 1, 5 * B))
        lo_w = max(32, n - B // 2)
        a = int(rng.integers(lo_w, n))
        cases.append((n, B, int(rng.random() < 0.7), (a, int(rng.integers(a, n + 1))),
                      int(rng.integers(0, 4))))
    return [oracle.keep_set(*c, prm) for c in cases]


def random_lists(rng, count):
    out = []
    for _ in range(count):
        m = int(rng.integers(1, 3000))
        steps = np.where(rng.random(m) < rng.random(), 1, rng.integers(1, 300, m))
        kept = np.cumsum(steps) - 1
        j0 = int(rng.integers(0, m + 1))
        kept[:j0] = np.arange(j0)
        kept[j0:] = np.maximum(kept[j0:], np.arange(j0, m) + 1)
        kept[j0:] = np.maximum.accumulate(kept[j0:] + np.arange(m - j0) * 0)
        for j in range(j0 + 1, m):                 # strictly increasing
            kept[j] = max(kept[j], kept[j - 1] + 1)
        out.append(kept.astype(np.int64))
    return out


def test_tiles_never_read_what_an_earlier_tile_wrote():
    rng = np.random.default_rng(3)
    for kept in keep_cases() + random_lists(rng, 200):
        cnt = len(kept)
        assert np.all(np.diff(kept) > 0) and np.all(kept >= np.arange(cnt))
        j0 = first_moved(kept)
        assert np.all(kept[j0:] > np.arange(j0, cnt))
        for T in (32, 64, 128, 170):
            for t0 in range(j0, cnt, T):
                t1 = min(t0 + T, cnt)
                # (b) rows read by later tiles lie above this tile's slots
                if t1 < cnt:
                    assert kept[t1] >= t1
                # (a) a slot of this tile is read only by this or an earlier tile
                readers = np.nonzero((kept >= t0) & (kept < t1))[0]
                assert readers.size == 0 or readers.max() < t1


def test_first_moved_search_matches_a_scan():
    rng = np.random.default_rng(5)
    lists = keep_cases() + random_lists(rng, 300) + [np.arange(0), np.arange(5), np.arange(1, 9)]
    for kept in lists:
        got, rounds = search32(kept, len(kept))
        assert got == first_moved(kept)
        assert rounds <= 4 or len(kept) > 32 ** 4


def test_kernel_source_order():
    with open(os.path.join(ROOT, "paper_2604_10044_gb300", "csrc", "lg_guard.cu")) as f:
        src = f.read()
    body = src[src.index("compact_kernel(lg_cache c"):]
    body = body[:body.index("// ------------------------------------------------------------------")]
    code = " ".join(re.sub(r"//[^\n]*", "", body).split())
    loop = code[code.index("for (int i = 0; i < n_tiles; ++i) {"):]
    order = ["cp_async_wait<kCompactStages - 2>();", "fence_proxy_async_smem();",
             "if (tid == 0) bulk_wait_read_all();", "__syncthreads();", "bulk_store(",
             "bulk_commit();", "const int p = i + kCompactStages - 1;",
             "if (p < n_tiles) gather(p);", "cp_async_commit();", "fetch_rows(p + 1);"]
    at = [loop.index(x) for x in order]
    assert at == sorted(at), order
    # the stage a gather refills is the one the previous tile's store has read
    S = int(re.search(r"kCompactStages = (\d+);", src).group(1))
    for i in range(3 * S):
        assert (i + S - 1) % S == (i - 1) % S
    # the search narrows to the first slot whose row moves
    assert "__ballot_sync(0xffffffffu, x < hi && kept[x] != x)" in code
    # barriers: two in the listing of the pruned sequences (one instead past 1024 sequences),
    # one per tile, one per item
    assert code.count("__syncthreads();") == 5, code.count("__syncthreads();")
