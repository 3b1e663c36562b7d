"""Pins for the oracle's trace statistics (Sec. 4.1-4.3, App. B), independent
of its code: a hand-worked example (tests/golden/trace_stats_example.json),
brute force in plain Python over token prefixes on tiny random traces, a
plain LRU simulation for the reachable reuses, a closed form for one growing
session, and the bookkeeping identities every trace satisfies."""
import json
import os
from collections import Counter, OrderedDict

import numpy as np
import pytest

import oracle
import tracegen

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _dense(sparse, shape):
    a = np.zeros(shape, dtype=np.uint64)
    for e in sparse:
        a[tuple(e[:-1])] = e[-1]
    return a


def _oracle_stats(tr, B, caps=None):
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    off = oracle.block_offsets(tr.req_tok_off, B)
    prev, _ = oracle.reuse(ids, D)
    sd = oracle.sd_fenwick(prev)
    st = oracle.trace_stats(ids, D, off, tr.req_ts_us, tr.req_session, tr.n_sessions, sd,
                            caps if caps is not None else [1])
    return st, ids, D, off, sd


def bit_length(x):
    return int(x).bit_length()


def bf_stats(requests, ts, sess, B, caps):
    """Every statistic straight from its definition: a block is its token
    prefix; each block keeps the list of (time, session) of its accesses."""
    per_req = Counter(sess)
    uses = {}  # prefix -> [(time, session), ...] in stream order
    stream = []
    for req, t, s in zip(requests, ts, sess):
        for k in range(len(req) // B):
            key = tuple(req[: B * (k + 1)])
            uses.setdefault(key, []).append((t, s))
            stream.append(key)
    out = {k: np.zeros(v, dtype=np.uint64) for k, v in oracle.STAT_SHAPES.items()}
    for key, acc in uses.items():
        sessions = {s for _, s in acc}
        if any(per_req[s] >= 2 for s in sessions):
            c = 0 if len(sessions) >= 2 else 1
        else:
            c = 2
        f = len(acc)
        life = acc[-1][0] - acc[0][0]
        out["blocks"][c] += 1
        out["accesses"][c] += f
        out["freq"][c, f if f < 256 else 0] += 1
        out["freq_log2"][c, bit_length(f)] += 1
        out["lifetime_us"][c, bit_length(life)] += 1
        out["lifetime_by_freq"][bit_length(f), bit_length(life)] += 1
        for (t0, _), (t1, _) in zip(acc[:-1], acc[1:]):
            out["reuse_us"][c, bit_length(t1 - t0)] += 1
            out["reuse_by_freq"][bit_length(f), bit_length(t1 - t0)] += 1
    # stack distance: 1 + distinct blocks strictly between two uses
    reach = [0] * len(caps)
    last = {}
    for i, key in enumerate(stream):
        if key in last:
            d = 1 + len(set(stream[last[key] + 1: i]))
            out["dist_log2"][bit_length(d)] += 1
            for g, C in enumerate(caps):
                reach[g] += d <= C
        last[key] = i
    times = {}
    for t, s in zip(ts, sess):
        times.setdefault(s, []).append(t)
    for s, tl in times.items():
        out["sess_requests"][bit_length(len(tl))] += 1
        out["sess_duration_us"][bit_length(max(tl) - min(tl))] += 1
    out.update(n_access=len(stream), n_distinct=len(uses), n_reuse=len(stream) - len(uses),
               n_sessions=len(times), n_multi_sessions=sum(1 for tl in times.values() if len(tl) >= 2))
    out["reach"] = np.array(reach, dtype=np.uint64)
    return out


def _same(a, b):
    for k in list(oracle.STAT_SHAPES) + list(oracle.STAT_SCALARS) + ["reach"]:
        assert np.array_equal(np.asarray(a[k]), np.asarray(b[k])), k


def test_trace_stats_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "trace_stats_example.json")))
    tr = tracegen.from_lists(g["requests"], ts=g["ts_us"], sessions=g["sessions"])
    B = g["block_size"]
    st, ids, D, off, sd = _oracle_stats(tr, B, g["capacities"])
    assert ids.tolist() == g["ids"]
    e = g["expect"]
    for k, shape in oracle.STAT_SHAPES.items():
        want = np.array(e[k], dtype=np.uint64) if len(shape) == 1 and k in ("blocks", "accesses") \
            else _dense(e[k], shape)
        assert np.array_equal(st[k], want), k
    assert st["reach"].tolist() == e["reach"]
    for k in oracle.STAT_SCALARS:
        assert st[k] == e[k], k


@pytest.mark.parametrize("seed", range(30))
def test_trace_stats_bruteforce_tiny(seed):
    rng = np.random.default_rng(5000 + seed)
    B = int(rng.integers(1, 4))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 9)), vocab=int(rng.integers(2, 5)))
    # arrival times with ties and long gaps; a few single-request sessions
    gaps = rng.choice([0, 1, 3, 1000, 7_000_000], size=tr.n_req)
    ts = np.cumsum(gaps).astype(np.int64)
    sess = tr.req_session.copy()
    reqs = [tr.tokens[int(a):int(b)].tolist() for a, b in zip(tr.req_tok_off[:-1], tr.req_tok_off[1:])]
    n_session = int(sess.max()) + 3  # two labels that no request uses
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    off = oracle.block_offsets(tr.req_tok_off, B)
    sd = oracle.sd_fenwick(oracle.reuse(ids, D)[0])
    caps = [1, 2, 3, 5, 8, 1000]
    st = oracle.trace_stats(ids, D, off, ts, sess, n_session, sd, caps)
    _same(st, bf_stats(reqs, ts.tolist(), sess.tolist(), B, caps))


def test_reach_is_plain_lru_hits():
    """A reuse is reachable within C blocks iff a plain LRU cache of C blocks
    (no prefix rule) hits on it (Mattson's inclusion)."""
    tr = tracegen.make(0).head(300)
    B = 16
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    off = oracle.block_offsets(tr.req_tok_off, B)
    sd = oracle.sd_fenwick(oracle.reuse(ids, D)[0])
    caps = [1, 7, 64, 500, 3000]
    st = oracle.trace_stats(ids, D, off, tr.req_ts_us, tr.req_session, tr.n_sessions, sd, caps)
    for C, got in zip(caps, st["reach"]):
        cache, hits = OrderedDict(), 0
        for x in ids.tolist():
            if x in cache:
                hits += 1
                cache.move_to_end(x)
            else:
                cache[x] = None
                if len(cache) > C:
                    cache.popitem(last=False)
        assert int(got) == hits, C


def test_growing_session_closed_form():
    """One session of k requests, request j holding the first j+1 tokens of
    one sequence (B = 1), arriving every g microseconds: block j is used by
    requests j .. k-1, so its frequency is k - j, its lifetime (k-1-j) g, and
    every reuse interval is g; all blocks are session history."""
    k, g = 23, 1500
    reqs = [list(range(1, j + 2)) for j in range(k)]
    tr = tracegen.from_lists(reqs, ts=[j * g for j in range(k)], sessions=[0] * k)
    st, ids, D, off, sd = _oracle_stats(tr, 1)
    assert D == k and st["n_reuse"] == k * (k - 1) // 2
    assert st["blocks"].tolist() == [0, k, 0]
    assert st["freq"][1, 1:k + 1].tolist() == [1] * k and int(st["freq"][1].sum()) == k
    assert st["reuse_us"][1, bit_length(g)] == k * (k - 1) // 2
    life = np.zeros(65, dtype=np.uint64)
    for j in range(k):
        life[bit_length((k - 1 - j) * g)] += 1
    assert np.array_equal(st["lifetime_us"][1], life)
    assert st["sess_requests"][bit_length(k)] == 1 and st["sess_duration_us"][bit_length((k - 1) * g)] == 1


def test_trace_stats_identities_conversational():
    """On the small conversational workload: the histograms partition the
    blocks, the accesses and the reuses; bins agree across views."""
    tr = tracegen.make(0)
    st, ids, D, off, sd = _oracle_stats(tr, 16, [1, 100, 10_000])
    N = ids.size
    assert st["n_access"] == N and st["n_distinct"] == D and st["n_reuse"] == N - D
    assert int(st["blocks"].sum()) == D and int(st["accesses"].sum()) == N
    for key in ("freq", "freq_log2", "lifetime_us"):
        assert np.array_equal(st[key].sum(axis=1), st["blocks"]), key
    assert np.array_equal(st["reuse_us"].sum(axis=1), st["accesses"] - st["blocks"])
    # a block used f times contributes f - 1 reuses to row bit_length(f)
    f = np.bincount(ids)
    rows = np.bincount([bit_length(x) for x in f], weights=f - 1, minlength=65).astype(np.uint64)
    assert np.array_equal(st["reuse_by_freq"].sum(axis=1), rows)
    assert np.array_equal(st["lifetime_by_freq"].sum(axis=1), st["freq_log2"].sum(axis=0))
    assert int(st["dist_log2"].sum()) == N - D and int(st["reach"][-1]) <= N - D
    assert int(st["sess_requests"].sum()) == st["n_sessions"] == np.unique(tr.req_session).size
    # a block used once has lifetime zero; single-turn blocks are used in single-request sessions only
    assert st["lifetime_by_freq"][1, 1:].sum() == 0
    counts = np.bincount(tr.req_session.astype(np.int64))
    assert st["n_multi_sessions"] == int((counts >= 2).sum())


def test_trace_stats_rejects_bad_input():
    tr = tracegen.from_lists([[1, 2], [1, 3]], ts=[5, 4], sessions=[0, 0])
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 1)
    off = oracle.block_offsets(tr.req_tok_off, 1)
    with pytest.raises(ValueError, match="decrease"):
        oracle.trace_stats(ids, D, off, tr.req_ts_us, tr.req_session, 1)
    with pytest.raises(ValueError, match="malformed"):
        oracle.trace_stats(ids, D, off, [4, 5], [0, 1], 1)
