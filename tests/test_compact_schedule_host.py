"""The barrier schedule of the in-place compaction (the index-gather of Sec. 5.3), on the CPU.

compact_kernel moves slot j <- row kept[j] (kept strictly increasing, kept[j] >= j) tile by
tile; the loads of tile i+1 are issued in iteration i, before that iteration's optional barrier
and its stores of tile i.  A barrier orders every load issued before it ahead of every store
after it.  The kernel takes the barrier of iteration i only when the lowest row read since the
last barrier lies below the tile's end.  Restated here and checked for safety: every store to
a slot s that some later index j reads (kept[j] = s) must be preceded by a barrier taken after
that load was issued.  The kernel's source is checked to contain the rule restated here.
"""
import os
import re

import numpy as np

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INF = 1 << 62


def schedule(kept, j0, cnt, T, rule="pending"):
    """iterations of the tile loop: list of (t0, barrier taken)"""
    out = []
    pend_row = kept[j0] if j0 < cnt else INF
    t0 = j0
    while t0 < cnt:
        t1 = t0 + T
        if rule == "pending":
            bar = pend_row < min(t1, cnt)
            if bar:
                jn = t1 + T
                pend_row = kept[jn] if jn < cnt else INF
        elif rule == "per_tile":          # kept[t0] >= t1 alone: not enough (see below)
            bar = kept[t0] < min(t1, cnt)
        else:
            bar = True
        out.append((t0, bar))
        t0 = t1
    return out


def first_moved(kept):
    j = 0
    while j < len(kept) and kept[j] == j:
        j += 1
    return j


def unsafe_pairs(kept, T, rule="pending"):
    """(j, s) pairs whose load of row s = kept[j] is not ordered before the store to slot s"""
    cnt = len(kept)
    j0 = first_moved(kept)
    sched = schedule(kept, j0, cnt, T, rule)
    bars = np.array([b for _, b in sched], dtype=bool)
    it = lambda j: (j - j0) // T          # iteration that stores slot j
    bad = []
    for j in range(j0, cnt):
        s = int(kept[j])
        if s >= cnt or s < j0:
            continue                      # row s is never overwritten by this stream
        if s == j:
            continue
        lo, hi = it(j) - 1, it(s)         # loads of tile it(j) are issued one iteration early
        lo = max(lo, 0)
        if not bars[lo:hi + 1].any():
            bad.append((j, s))
    return bad, int(bars.sum()), len(sched)


def keep_cases():
    prm = oracle.params()
    rng = np.random.default_rng(7)
    cases = [(8193, 4096, 0, (0, 0), 0), (131073, 32768, 0, (0, 0), 0),
             (131073, 32768, 1, (114689, 131073), 0), (32769, 8192, 1, (32000, 32600), 1),
             (5000, 4096, 1, (4900, 4940), 0), (5000, 4096, 1, (4800, 4864), 0),
             (5000, 4096, 1, (4800, 4863), 2), (5000, 4096, 1, (4800, 4865), 3),
             (4200, 4096, 0, (0, 0), 0), (4097, 4096, 0, (0, 0), 0)]
    for _ in range(60):
        B = int(rng.choice([256, 1024, 4096, 8192]))
        n = int(rng.integers(B + 1, 5 * B))
        lo_w = max(32, n - B // 2)
        a = int(rng.integers(lo_w, n))
        cases.append((n, B, int(rng.random() < 0.7), (a, int(rng.integers(a, n + 1))),
                      int(rng.integers(0, 4))))
    return [(c, oracle.keep_set(*c, prm)) for c in cases]


def random_lists(rng, count):
    """increasing lists with kept[j] >= j mixing dense stretches (steps of 1) and gaps"""
    out = []
    for _ in range(count):
        m = int(rng.integers(50, 3000))
        steps = np.where(rng.random(m) < rng.random(), 1, rng.integers(1, 300, m))
        kept = np.cumsum(steps) - 1 + int(rng.integers(0, 5))
        kept = np.maximum(kept, np.arange(m))
        out.append(kept.astype(np.int64))
    return out


def test_pending_rule_orders_every_load_before_its_slot_is_written():
    rng = np.random.default_rng(11)
    lists = [k for _, k in keep_cases()] + random_lists(rng, 300)
    for kept in lists:
        for T in (16, 32, 64, 128):
            bad, _, _ = unsafe_pairs(kept, T)
            assert not bad, (T, bad[:3])


def test_sparse_lattice_takes_few_barriers():
    """a budget cut of a long cache (every 4th row kept) takes a barrier only where the tiles
    catch up with the rows still pending: a handful per stream instead of one per tile"""
    prm = oracle.params()
    kept = oracle.keep_set(131073, 32768, 0, (0, 0), 0, prm)
    _, n_bar, n_it = unsafe_pairs(kept, 64)
    assert n_it == 511 and n_bar <= 12, (n_bar, n_it)
    # the dense recent block of the 8192-row budget cut keeps a constant offset of 4161 rows
    kept = oracle.keep_set(8193, 4096, 0, (0, 0), 0, prm)
    _, n_bar, n_it = unsafe_pairs(kept, 64)
    assert n_bar <= n_it // 4, (n_bar, n_it)
    # a short removed span (40 rows < one tile) leaves every later tile overlapping its rows
    kept = oracle.keep_set(5000, 4096, 1, (4900, 4940), 0, prm)
    bad, n_bar, n_it = unsafe_pairs(kept, 64)
    assert not bad and n_bar >= 1


def test_per_tile_test_alone_is_unsafe():
    """kept[t0] >= t1 says only that the tile's own rows lie above its slots; without a barrier a
    warp may store the next tile's slots while another still loads this tile's rows there"""
    kept = np.concatenate([np.arange(0, 10), np.arange(74, 74 + 400)])
    bad, _, _ = unsafe_pairs(kept, 64, rule="per_tile")
    assert bad
    assert not unsafe_pairs(kept, 64)[0]


def test_kernel_source_has_the_rule():
    with open(os.path.join(ROOT, "paper_2604_10044_gb300", "csrc", "lg_guard.cu")) as f:
        src = f.read()
    body = src[src.index("compact_kernel(lg_cache c"):]
    body = body[:body.index("// ------------------------------------------------------------------")]
    code = re.sub(r"//[^\n]*", "", body)
    code = " ".join(code.split())
    assert "int pend_row = j0 < cnt ? kept[j0] : INT_MAX;" in code
    assert "if (t1 < cnt) load_tile(nxt, t1); if (pend_row < min(t1, cnt)) { __syncthreads();" \
        in code
    assert "const int jn = t1 + rows_per_tile; pend_row = jn < cnt ? kept[jn] : INT_MAX;" in code
    # exactly one barrier inside the tile loop (the conditional one)
    loop = code[code.index("for (int t0 = j0;"):code.index("cur[k] = nxt[k]; }")]
    assert loop.count("__syncthreads()") == 1
