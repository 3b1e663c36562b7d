"""Pins for the CPU oracle, independent of the oracle's own code.

Each check compares the oracle with something the paper or mathematics fixes:
a hand-worked example (tests/golden/worked_example.json), brute force on tiny
random traces written here in plain Python (prefix tuples, window sets,
OrderedDict LRU), closed forms, and invariants of LRU stack distances.
"""
import json
import os
from collections import OrderedDict

import numpy as np
import pytest

import oracle
import tracegen

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
NONE = oracle.NONE


def _none(v):
    return [NONE if x is None else x for x in v]


# ---------------------------------------------------------------- brute force
def bf_ids(requests, B):
    """Block identity = the whole token prefix up to the block's end (Sec. 2.2)."""
    table, ids, req_blk_off = {}, [], [0]
    for req in requests:
        n = len(req) // B
        for k in range(n):
            key = tuple(req[: B * (k + 1)])
            if key not in table:
                table[key] = len(table)
            ids.append(table[key])
        req_blk_off.append(req_blk_off[-1] + n)
    return ids, len(table), req_blk_off


def bf_prev_next(ids):
    n = len(ids)
    prev = [NONE] * n
    nxt = [NONE] * n
    for i in range(n):
        for j in range(i - 1, -1, -1):
            if ids[j] == ids[i]:
                prev[i] = j
                break
        for j in range(i + 1, n):
            if ids[j] == ids[i]:
                nxt[i] = j
                break
    return prev, nxt


def bf_sd(ids):
    """1 + number of distinct blocks strictly between two accesses of a block."""
    sd, last = [], {}
    for i, x in enumerate(ids):
        if x in last:
            sd.append(1 + len(set(ids[last[x] + 1: i])))
        else:
            sd.append(NONE)
        last[x] = i
    return sd


def bf_cost(k, B, kind, f_lin, f_attn):
    if kind == 0:
        return 1
    lin = B * f_lin if kind == 1 else 0
    return lin + sum(f_attn * (t + 1) for t in range(B * k, B * k + B))


def bf_lru(ids, req_blk_off, B, C, kind, f_lin, f_attn):
    cache = OrderedDict()
    hits = saved = 0
    for r in range(len(req_blk_off) - 1):
        ok = True
        for k in range(req_blk_off[r + 1] - req_blk_off[r]):
            x = ids[req_blk_off[r] + k]
            resident = x in cache
            if resident:
                cache.move_to_end(x)
            else:
                cache[x] = True
                if len(cache) > C:
                    cache.popitem(last=False)
            ok = ok and resident
            if ok:
                hits += 1
                saved += bf_cost(k, B, kind, f_lin, f_attn)
    return hits, saved


# ---------------------------------------------------------------- worked example
def test_worked_example_exact():
    g = json.load(open(os.path.join(GOLDEN, "worked_example.json")))
    tr = tracegen.from_lists(g["requests"])
    B = g["block_size"]
    off = oracle.block_offsets(tr.req_tok_off, B)
    assert off.tolist() == g["req_blk_off"]
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    assert ids.tolist() == g["ids"] and D == g["n_distinct"]
    prev, nxt = oracle.reuse(ids, D)
    assert prev.tolist() == _none(g["prev"])
    assert nxt.tolist() == _none(g["next"])
    assert oracle.sd_fenwick(prev).tolist() == _none(g["sd"])
    assert oracle.sd_mattson(ids).tolist() == _none(g["sd"])
    cm = g["cost_model"]
    hits, saved, total = oracle.lru_curves(ids, off, B, g["capacities"], cm["kind"], cm["f_lin"], cm["f_attn"])
    assert hits == g["hits"]
    assert saved == g["saved"]
    assert total == g["total_cost"]


# ---------------------------------------------------------------- random tiny traces
@pytest.mark.parametrize("seed", range(40))
def test_bruteforce_tiny(seed):
    rng = np.random.default_rng(1000 + seed)
    B = int(rng.integers(1, 5))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 8)), vocab=int(rng.integers(2, 5)))
    reqs = [tr.tokens[int(a):int(b)].tolist() for a, b in zip(tr.req_tok_off[:-1], tr.req_tok_off[1:])]
    ids_bf, D_bf, off_bf = bf_ids(reqs, B)

    off = oracle.block_offsets(tr.req_tok_off, B)
    assert off.tolist() == off_bf
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    assert ids.tolist() == ids_bf and D == D_bf
    prev, nxt = oracle.reuse(ids, D)
    p_bf, n_bf = bf_prev_next(ids_bf)
    assert prev.tolist() == p_bf and nxt.tolist() == n_bf
    sd_bf = bf_sd(ids_bf)
    assert oracle.sd_fenwick(prev).tolist() == sd_bf
    assert oracle.sd_mattson(ids).tolist() == sd_bf

    kind = int(rng.integers(0, 3))
    f_lin, f_attn = int(rng.integers(0, 1000)), int(rng.integers(0, 1000))
    caps = list(range(1, D + 2))
    hits, saved, total = oracle.lru_curves(ids, off, B, caps, kind, f_lin, f_attn)
    for C, h, s in zip(caps, hits, saved):
        assert (h, s) == bf_lru(ids_bf, off_bf, B, C, kind, f_lin, f_attn), C
    assert total == sum(bf_cost(k, B, kind, f_lin, f_attn)
                        for r in range(len(off_bf) - 1) for k in range(off_bf[r + 1] - off_bf[r]))


def test_empty_and_short_requests():
    tr = tracegen.from_lists([[], [1], [1, 2, 3], [], [1, 2, 3, 4]])
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 2)
    assert ids.tolist() == [0, 0, 1] and D == 2
    assert oracle.block_offsets(tr.req_tok_off, 2).tolist() == [0, 0, 0, 1, 1, 3]
    e = tracegen.from_lists([])
    ids, D = oracle.block_ids(e.tokens, e.req_tok_off, 16)
    assert ids.size == 0 and D == 0
    hits, saved, total = oracle.lru_curves(ids, np.zeros(1, np.uint64), 16, [1, 5])
    assert hits == [0, 0] and saved == [0, 0] and total == 0


# ---------------------------------------------------------------- invariants
@pytest.fixture(scope="module")
def small_conv():
    tr = tracegen.make(0).head(400)
    B = 16
    off = oracle.block_offsets(tr.req_tok_off, B)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    prev, nxt = oracle.reuse(ids, D)
    sd = oracle.sd_fenwick(prev)
    return tr, B, off, ids, D, prev, nxt, sd


def _running_max(sd, off):
    e = sd.astype(np.int64).copy()
    e[sd == NONE] = 1 << 40
    for r in range(len(off) - 1):
        a, b = int(off[r]), int(off[r + 1])
        if b > a:
            e[a:b] = np.maximum.accumulate(e[a:b])
    return e


def test_mattson_inclusion_and_monotone(small_conv):
    """Direct simulation at every capacity equals the stack-distance threshold
    count (Mattson et al. 1970), and curves are non-decreasing in C."""
    tr, B, off, ids, D, prev, nxt, sd = small_conv
    caps = tracegen.capacity_grid(1, D + 5, 24)
    hits, saved, total = oracle.lru_curves(ids, off, B, caps)
    e = _running_max(sd, off)
    k = np.concatenate([np.arange(int(off[r + 1] - off[r])) for r in range(len(off) - 1)])
    for C, h, s in zip(caps, hits, saved):
        mask = e <= int(C)
        assert h == int(mask.sum())
        assert s == sum(bf_cost(int(x), B, 1, oracle.F_LIN, oracle.F_ATTN) for x in k[mask])
    assert all(a <= b for a, b in zip(hits, hits[1:]))
    assert all(a <= b for a, b in zip(saved, saved[1:]))
    # cold identity: at a capacity above D every non-cold access hits
    assert hits[-1] == ids.size - D


def test_running_max_is_noop_rootfirst(small_conv):
    """Root-first replay: a non-cold block's distance is never below its
    parent's, so the per-request running max leaves distances unchanged."""
    tr, B, off, ids, D, prev, nxt, sd = small_conv
    e = _running_max(sd, off)
    s = sd.astype(np.int64)
    s[sd == NONE] = 1 << 40
    assert np.array_equal(e, s)


def test_next_prev_consistency(small_conv):
    tr, B, off, ids, D, prev, nxt, sd = small_conv
    warm = prev != NONE
    assert np.array_equal(nxt[prev[warm]], np.nonzero(warm)[0].astype(np.uint32))
    assert int((nxt == NONE).sum()) == D and int((prev == NONE).sum()) == D
    assert np.all(ids[prev[warm]] == ids[warm])


def test_single_session_closed_form():
    """One session whose requests each extend the previous one: every re-read
    block has distance n_{t-1} (the previous request's block count), so
    hits(C) = sum_t n_{t-1} [n_{t-1} <= C]."""
    rng = np.random.default_rng(7)
    B = 4
    ctx, reqs = [], []
    for _ in range(9):
        ctx = ctx + [int(x) for x in rng.integers(0, 1000, int(rng.integers(1, 30)))]
        reqs.append(list(ctx))
    tr = tracegen.from_lists(reqs)
    off = oracle.block_offsets(tr.req_tok_off, B)
    n = np.diff(off).astype(int)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    prev, _ = oracle.reuse(ids, D)
    sd = oracle.sd_fenwick(prev)
    for t in range(1, len(n)):
        a = int(off[t])
        reread = min(n[t - 1], n[t])
        assert sd[a:a + reread].tolist() == [n[t - 1]] * reread
    caps = list(range(1, int(n.max()) + 3))
    hits, saved, _ = oracle.lru_curves(ids, off, B, caps, 2, 0, 3)
    for C, h, s in zip(caps, hits, saved):
        exp_h = sum(min(n[t - 1], n[t]) for t in range(1, len(n)) if n[t - 1] <= C)
        exp_s = sum(3 * sum(t_ + 1 for t_ in range(B * k, B * k + B))
                    for t in range(1, len(n)) if n[t - 1] <= C for k in range(min(n[t - 1], n[t])))
        assert (h, s) == (exp_h, exp_s), C


def test_total_cost_closed_form(small_conv):
    """Sum of cost(k) over each request's blocks in closed form:
    n*B*f_lin + f_attn*(B^2 n(n-1)/2 + n B(B+1)/2)."""
    tr, B, off, ids, D, prev, nxt, sd = small_conv
    _, _, total = oracle.lru_curves(ids, off, B, [1])
    exp = 0
    for r in range(len(off) - 1):
        n = int(off[r + 1] - off[r])
        exp += n * B * oracle.F_LIN + oracle.F_ATTN * (B * B * n * (n - 1) // 2 + n * B * (B + 1) // 2)
    assert total == exp


def test_scan_longer_than_capacity_never_hits():
    """A cyclic scan over more distinct blocks than the cache holds misses
    every time under LRU."""
    reqs = [[i] for i in range(10)] * 3
    tr = tracegen.from_lists(reqs)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 1)
    off = oracle.block_offsets(tr.req_tok_off, 1)
    hits, _, _ = oracle.lru_curves(ids, off, 1, [9, 10], 0)
    assert hits == [0, 20]


# ---------------------------------------------------------------- prefix hash
P61 = (1 << 61) - 1


def _splitmix(seed, n):
    z = (seed + (n + 1) * 0x9E3779B97F4A7C15) & (2**64 - 1)
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & (2**64 - 1)
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & (2**64 - 1)
    return z ^ (z >> 31)


def test_splitmix_published_vector():
    """SplitMix64 from state 0: the first outputs of the published generator."""
    assert _splitmix(0, 0) == 0xE220A8397B1DCDAF
    assert _splitmix(0, 1) == 0x6E789E6AA1B965F4
    assert _splitmix(0, 2) == 0x06C45D188009454F
    lib = tracegen._load()
    assert [lib.tg_sm64_at(0, n) for n in range(3)] == [_splitmix(0, n) for n in range(3)]


@pytest.mark.parametrize("seed", [0, 1, 12345, 2**63 + 7])
def test_prefix_hash_polynomial(seed):
    """Keys equal sum_t (tok_t + 1) u^(t+1) mod 2^61 - 1 over the block's
    whole prefix at the two seeded bases, evaluated with Python integers from
    the sum definition (tokens up to 2^32 - 1 included)."""
    tr = tracegen.tiny(seed % 1000, n_sessions=4, vocab=2**32 - 1 if seed & 1 else 5)
    B = 3
    keys = oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, seed)
    u = [2 + _splitmix(seed, b) % (P61 - 3) for b in range(2)]
    i = 0
    for a, b in zip(tr.req_tok_off[:-1], tr.req_tok_off[1:]):
        toks = [int(x) for x in tr.tokens[int(a):int(b)]]
        for k in range(len(toks) // B):
            m = B * (k + 1)
            for base in range(2):
                h = sum((toks[t] + 1) * pow(u[base], t + 1, P61) for t in range(m))
                assert int(keys[i, base]) == h % P61
            i += 1
    assert i == keys.shape[0]


def test_prefix_hash_separates_lengths():
    """Coefficients tok + 1 >= 1 keep a prefix and its zero-extension apart."""
    tr = tracegen.from_lists([[0, 0], [0, 0, 0, 0]])
    keys = oracle.prefix_hash(tr.tokens, tr.req_tok_off, 2, 99)
    assert not np.array_equal(keys[0], keys[2])
    assert np.array_equal(keys[0], keys[1])


# ---------------------------------------------------------------- curves by inclusion
@pytest.mark.parametrize("seed", range(12))
def test_curves_from_dist_bruteforce(seed):
    """orc_curves_from_dist (the inclusion route the GPU takes) against the
    plain-Python OrderedDict LRU at every capacity from 1 to D + 2, with
    distances from window sets, under all three cost kinds."""
    tr = tracegen.tiny(500 + seed, n_sessions=5, vocab=2)
    B = 1 + seed % 3
    reqs = [list(tr.tokens[int(tr.req_tok_off[r]):int(tr.req_tok_off[r + 1])]) for r in range(tr.n_req)]
    ids, D, off = bf_ids(reqs, B)
    sd = np.asarray(bf_sd(ids), dtype=np.uint32)
    caps = np.arange(1, D + 3, dtype=np.uint64)
    for kind, f_lin, f_attn in ((0, 0, 0), (1, 5, 3), (2, 0, 7)):
        hits, saved = oracle.curves_from_dist(sd, off, B, caps, kind, f_lin, f_attn)
        for C, h, s in zip(caps, hits, saved):
            assert (h, s) == bf_lru(ids, off, B, int(C), kind, f_lin, f_attn)


def test_curves_from_dist_equals_direct_lru(small_conv):
    """On the tiny conversational workload: the inclusion route equals the
    oracle's direct per-capacity LRU simulation (Mattson inclusion), hits and
    128-bit compute saved, on a grid that includes capacities past D."""
    tr, B, off, ids, D, prev, nxt, sd = small_conv
    caps = tracegen.capacity_grid(1, D + 5, 20)
    hits, saved, _ = oracle.lru_curves(ids, off, B, caps)
    h2, s2 = oracle.curves_from_dist(sd, off, B, caps)
    assert hits == h2 and saved == s2


def test_curves_from_dist_rejects_bad_grid():
    with pytest.raises(ValueError):
        oracle.curves_from_dist(np.zeros(1, np.uint32), np.array([0, 1], np.uint64), 1, np.array([3, 3], np.uint64))
    with pytest.raises(ValueError):
        oracle.curves_from_dist(np.zeros(1, np.uint32), np.array([0, 1], np.uint64), 1, np.array([0], np.uint64))
