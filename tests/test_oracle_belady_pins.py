"""Pins for the oracle's Belady curves (orc_belady_curves), independent of
its code.

Belady's MIN (Belady 1966) is the paper's offline ceiling (Sec. 3.2).  The
oracle simulates it directly: on a miss with a full cache, evict the resident
block (not the one just brought in) whose next access is farthest.  Checked
here against:
  * exhaustive search over every eviction choice on tiny traces: MIN's raw
    hit count is the largest any demand-paging policy reaches (Belady's
    theorem; Mattson et al. 1970);
  * a plain-Python MIN that finds next accesses by scanning the trace forward,
    with the prefix rule of Sec. 2.2 and the three cost kinds;
  * the interval view: a reuse of a block hits iff it is kept from its
    previous access, and the hits are the largest set of reuse intervals in
    which no access time lies strictly inside more than C - 1 of them, built
    greedily by end time with best-fit tracks (Carlisle and Lloyd 1995);
  * theorems: raw hits at least LRU's at every C, monotone in C (OPT is a
    stack algorithm), only immediate repeats hit at C = 1 (the same as LRU),
    N - D hits once nothing is evicted.
"""
import itertools
import random

import numpy as np
import pytest

import oracle
import tracegen

NONE = oracle.NONE


def prefix_ids(requests, B):
    table, ids, off = {}, [], [0]
    for req in requests:
        n = len(req) // B
        for k in range(n):
            key = tuple(req[: B * (k + 1)])
            ids.append(table.setdefault(key, len(table)))
        off.append(off[-1] + n)
    return ids, len(table), off


def cost(k, B, kind, f_lin, f_attn):
    if kind == 0:
        return 1
    return (B * f_lin if kind == 1 else 0) + sum(f_attn * (t + 1) for t in range(B * k, B * k + B))


def py_min(ids, off, B, C, kind=1, f_lin=5, f_attn=3):
    """MIN with next accesses found by scanning forward; prefix-counted hits,
    compute saved and raw hits."""
    n = len(ids)
    cache = set()
    hits = saved = raw = 0

    def next_use(x, i):
        for j in range(i + 1, n):
            if ids[j] == x:
                return j
        return float("inf")

    for r in range(len(off) - 1):
        ok = True
        for k in range(off[r + 1] - off[r]):
            i = off[r] + k
            x = ids[i]
            res = x in cache
            if not res:
                cache.add(x)
                if len(cache) > C:
                    others = [y for y in cache if y != x]
                    far = max(next_use(y, i) for y in others)
                    cache.remove(next(y for y in others if next_use(y, i) == far))
            raw += res
            ok = ok and res
            if ok:
                hits += 1
                saved += cost(k, B, kind, f_lin, f_attn)
    return hits, saved, raw


def greedy_hit_set(ids, C):
    """Reuse intervals by end time, best-fit tracks: the set of hitting accesses."""
    last, prev = {}, []
    for i, x in enumerate(ids):
        prev.append(last.get(x))
        last[x] = i
    tracks = [float("-inf")] * (C - 1)
    hit = [False] * len(ids)
    for i, p in enumerate(prev):
        if p is None:
            continue
        if p == i - 1:
            hit[i] = True
            continue
        fits = [f for f in tracks if f <= p]
        if fits:
            tracks.remove(max(fits))
            tracks.append(i - 1)
            hit[i] = True
    return hit


def best_possible_raw_hits(ids, C):
    """Every demand-paging policy: at each miss with a full cache, try every victim."""
    best = 0

    def go(i, cache, h):
        nonlocal best
        if i == len(ids):
            best = max(best, h)
            return
        if h + (len(ids) - i) <= best:
            return
        x = ids[i]
        if x in cache:
            go(i + 1, cache, h + 1)
            return
        if len(cache) < C:
            go(i + 1, cache | {x}, h)
            return
        for v in cache:
            go(i + 1, (cache - {v}) | {x}, h)

    go(0, frozenset(), 0)
    return best


@pytest.mark.parametrize("seed", range(40))
def test_exhaustive_optimum(seed):
    rnd = random.Random(seed)
    n, V = rnd.randint(1, 11), rnd.randint(1, 5)
    ids = [rnd.randrange(V) for _ in range(n)]
    off = np.array([0, n], dtype=np.uint64)
    D = len(set(ids))
    caps = np.arange(1, D + 2, dtype=np.uint64)
    _, _, raw = oracle.belady_curves(np.asarray(ids, np.uint32), off, 1, caps, 0)
    for C, r in zip(caps, raw):
        assert r == best_possible_raw_hits(ids, int(C)), (ids, int(C))


@pytest.mark.parametrize("seed", range(24))
def test_plain_python_min_with_prefix_rule(seed):
    tr = tracegen.tiny(700 + seed, n_sessions=5, vocab=2, max_seg=6)
    B = 1 + seed % 3
    reqs = [list(tr.tokens[int(tr.req_tok_off[r]):int(tr.req_tok_off[r + 1])]) for r in range(tr.n_req)]
    ids, D, off = prefix_ids(reqs, B)
    caps = np.arange(1, D + 2, dtype=np.uint64)
    for kind, f_lin, f_attn in ((0, 0, 0), (1, 5, 3), (2, 0, 7)):
        h, s, raw = oracle.belady_curves(np.asarray(ids, np.uint32), np.asarray(off, np.uint64), B, caps, kind,
                                         f_lin, f_attn)
        for g, C in enumerate(caps):
            assert (h[g], s[g], raw[g]) == py_min(ids, off, B, int(C), kind, f_lin, f_attn), (kind, int(C))


@pytest.mark.parametrize("seed", range(16))
def test_interval_greedy_hit_set(seed):
    """The prefix-counted hits follow from the interval view's hit set."""
    tr = tracegen.tiny(900 + seed, n_sessions=7, vocab=3, max_seg=9)
    B = 1 + seed % 2
    reqs = [list(tr.tokens[int(tr.req_tok_off[r]):int(tr.req_tok_off[r + 1])]) for r in range(tr.n_req)]
    ids, D, off = prefix_ids(reqs, B)
    caps = np.arange(1, D + 2, dtype=np.uint64)
    h, s, raw = oracle.belady_curves(np.asarray(ids, np.uint32), np.asarray(off, np.uint64), B, caps, 0)
    for g, C in enumerate(caps):
        hit = greedy_hit_set(ids, int(C))
        assert raw[g] == sum(hit)
        counted = 0
        for r in range(len(off) - 1):
            for k in range(off[r + 1] - off[r]):
                if not hit[off[r] + k]:
                    break
                counted += 1
        assert h[g] == counted


@pytest.fixture(scope="module")
def small_conv():
    tr = tracegen.make(0).head(400)
    B = 16
    off = oracle.block_offsets(tr.req_tok_off, B)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    return ids, D, off


def test_theorems_on_the_tiny_workload(small_conv):
    ids, D, off = small_conv
    caps = np.unique(np.concatenate([[1, 2, 3], tracegen.capacity_grid(4, D + 3, 20)])).astype(np.uint64)
    h, s, raw = oracle.belady_curves(ids, off, 16, caps)
    lh, ls, _ = oracle.lru_curves(ids, off, 16, caps)
    prev, _ = oracle.reuse(ids, D)
    N = ids.size
    for g in range(len(caps)):
        assert raw[g] >= lh[g]  # LRU's prefix-counted hits equal its raw hits
        assert h[g] <= raw[g]
    assert all(a <= b for a, b in zip(h, h[1:])) and all(a <= b for a, b in zip(raw, raw[1:]))
    assert all(a <= b for a, b in zip(s, s[1:]))
    # C = 1: only a block accessed again right away can hit
    imm = int(np.sum(prev[1:].astype(np.int64) == np.arange(N - 1)))
    assert raw[0] == imm and h[0] == lh[0]
    # nothing evicted: every reuse hits, and the prefix rule removes nothing
    assert caps[-1] >= D and h[-1] == raw[-1] == N - D


def test_rejects_capacity_zero():
    with pytest.raises(ValueError):
        oracle.belady_curves(np.zeros(1, np.uint32), np.array([0, 1], np.uint64), 1, np.array([0], np.uint64))
