"""Pins for the oracle's session-level LRU curves (orc_session_lru_curves),
independent of its code: the hand-worked example
tests/golden/session_lru_example.json, a plain-Python brute force with other
data structures (recency as a Python list of sessions, ownership recomputed
from per-session sets) on tiny random traces at every capacity and cost
kind, and identities: N - D hits once nothing is evicted, and every reuse
hits when sessions are disjoint, one after another, each fitting in C."""
import json
import os

import numpy as np
import pytest

import oracle
import tracegen

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def prefix_ids(requests, B):
    table, ids, off = {}, [], [0]
    for req in requests:
        n = len(req) // B
        for k in range(n):
            ids.append(table.setdefault(tuple(req[: B * (k + 1)]), len(table)))
        off.append(off[-1] + n)
    return ids, len(table), off


def cost(k, B, kind, f_lin, f_attn):
    if kind == 0:
        return 1
    return (B * f_lin if kind == 1 else 0) + sum(f_attn * (t + 1) for t in range(B * k, B * k + B))


def brute_session_lru(ids, off, sessions, B, C, kind=0, f_lin=0, f_attn=0):
    recency = []   # sessions, least recently touched first
    held = {}      # session -> set of blocks it brought in and still holds
    hits = saved = 0
    for r in range(len(off) - 1):
        s = sessions[r]
        if s in recency:
            recency.remove(s)
        recency.append(s)
        ok = True
        for k in range(off[r + 1] - off[r]):
            x = ids[off[r] + k]
            res = any(x in blocks for blocks in held.values())
            if not res:
                held.setdefault(s, set()).add(x)
                while sum(len(b) for b in held.values()) > C:
                    others = [t for t in recency if t != s and held.get(t)]
                    if others:
                        held[others[0]] = set()
                    else:
                        held[s] = {x}
            ok = ok and res
            if ok:
                hits += 1
                saved += cost(k, B, kind, f_lin, f_attn)
    return hits, saved


def test_hand_worked_example():
    with open(os.path.join(GOLDEN, "session_lru_example.json")) as f:
        g = json.load(f)
    tr = tracegen.from_lists(g["requests"], sessions=g["sessions"])
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 1)
    assert ids.tolist() == g["block_ids"]
    off = oracle.block_offsets(tr.req_tok_off, 1)
    h, s = oracle.session_lru_curves(ids, off, np.asarray(g["sessions"], np.uint32), 2, 1,
                                     np.asarray(g["capacities"], np.uint64), oracle.COST_UNIFORM)
    assert h == g["hits"] and s == g["hits"]


@pytest.mark.parametrize("seed", range(40))
def test_bruteforce_tiny(seed):
    rng = np.random.default_rng(4000 + seed)
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 7)), max_turns=5, vocab=int(rng.integers(2, 4)),
                       max_seg=int(rng.integers(2, 8)))
    B = int(rng.integers(1, 4))
    reqs = [list(tr.tokens[int(tr.req_tok_off[r]):int(tr.req_tok_off[r + 1])]) for r in range(tr.n_req)]
    ids, D, off = prefix_ids(reqs, B)
    ses = [int(x) for x in tr.req_session]
    S = max(ses) + 1 if ses else 1
    caps = np.arange(1, D + 3, dtype=np.uint64)
    for kind, f_lin, f_attn in ((0, 0, 0), (1, 5, 3), (2, 0, 7)):
        h, s = oracle.session_lru_curves(np.asarray(ids, np.uint32), np.asarray(off, np.uint64),
                                         np.asarray(ses, np.uint32), S, B, caps, kind, f_lin, f_attn)
        for g, C in enumerate(caps):
            assert (h[g], s[g]) == brute_session_lru(ids, off, ses, B, int(C), kind, f_lin, f_attn), (kind, int(C))


def test_nothing_evicted_and_disjoint_sequential_sessions():
    tr = tracegen.make(0).head(300)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    off = oracle.block_offsets(tr.req_tok_off, 16)
    ses = tr.req_session.astype(np.uint32)
    h, _ = oracle.session_lru_curves(ids, off, ses, tr.n_sessions, 16, np.array([D, D + 10], np.uint64))
    assert h == [ids.size - D] * 2
    # disjoint sessions, one after another, each fitting in C: every reuse hits
    reqs, sess = [], []
    for s in range(5):
        base = [100 * s + t for t in range(3)]
        for turn in range(4):
            reqs.append(base + [100 * s + 10 + t for t in range(turn)])
            sess.append(s)
    tr2 = tracegen.from_lists(reqs, sessions=sess)
    ids2, D2 = oracle.block_ids(tr2.tokens, tr2.req_tok_off, 1)
    off2 = oracle.block_offsets(tr2.req_tok_off, 1)
    h2, _ = oracle.session_lru_curves(ids2, off2, np.asarray(sess, np.uint32), 5, 1, np.array([6, 7], np.uint64))
    assert h2 == [ids2.size - D2] * 2


def test_rejects_bad_input():
    with pytest.raises(ValueError):
        oracle.session_lru_curves(np.zeros(1, np.uint32), np.array([0, 1], np.uint64), np.array([3], np.uint32), 3,
                                  1, np.array([1], np.uint64))
    with pytest.raises(ValueError):
        oracle.session_lru_curves(np.zeros(1, np.uint32), np.array([0, 1], np.uint64), np.array([0], np.uint32), 1,
                                  1, np.array([0], np.uint64))
