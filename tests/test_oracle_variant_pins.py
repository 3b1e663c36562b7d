"""Pins for the oracle's semantics variants (Sec. 3.1: the paper's simulator
keeps a whole request resident and makes room for it up front; engines
differ in the order they touch a request's blocks), independent of the
oracle's code: brute force in plain Python (OrderedDict LRU per capacity,
list-based LRU stacks), the hot path's own semantics as the special case
(root-first, per block), Mattson inclusion, and closed forms for one growing
session under every variant."""
from collections import OrderedDict

import numpy as np
import pytest

import oracle
import tracegen

NONE = oracle.NONE
VARIANTS = [(o, r) for o in (oracle.ROOT_FIRST, oracle.LEAF_FIRST) for r in (oracle.RES_BLOCK, oracle.RES_REQUEST)]


def bf_requests(requests, B):
    """Block identity = the whole token prefix (Sec. 2.2); one list per request."""
    return [[tuple(req[: B * (k + 1)]) for k in range(len(req) // B)] for req in requests]


def bf_cost(k, B, kind, f_lin, f_attn):
    if kind == 0:
        return 1
    attn = f_attn * sum(t + 1 for t in range(B * k, B * k + B))
    return attn + (B * f_lin if kind == 1 else 0)


def bf_lru(blocks, B, C, order, residency, kind, f_lin, f_attn):
    cache = OrderedDict()  # last = most recent
    hits = saved = 0

    def touch(x):
        if x in cache:
            cache.move_to_end(x)
        else:
            cache[x] = None
            if len(cache) > C:
                cache.popitem(last=False)

    for req in blocks:
        seq = list(range(len(req))) if order == oracle.ROOT_FIRST else list(range(len(req)))[::-1]
        found = [x in cache for x in req] if residency == oracle.RES_REQUEST else [None] * len(req)
        for k in seq:
            if residency == oracle.RES_BLOCK:
                found[k] = req[k] in cache
            touch(req[k])
        for k in range(len(req)):
            if not found[k]:
                break
            hits += 1
            saved += bf_cost(k, B, kind, f_lin, f_attn)
    return hits, saved


def bf_sd(blocks, order, residency):
    """Depth in the recency stack (1 = most recent) when looked up."""
    stack, out = [], []  # stack[0] = most recent
    for req in blocks:
        seq = list(range(len(req))) if order == oracle.ROOT_FIRST else list(range(len(req)))[::-1]
        d = [None] * len(req)
        if residency == oracle.RES_REQUEST:
            d = [stack.index(x) + 1 if x in stack else NONE for x in req]
        for k in seq:
            if residency == oracle.RES_BLOCK:
                d[k] = stack.index(req[k]) + 1 if req[k] in stack else NONE
            if req[k] in stack:
                stack.remove(req[k])
            stack.insert(0, req[k])
        out.extend(d)
    return out


def _setup(tr, B):
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    off = oracle.block_offsets(tr.req_tok_off, B)
    return ids, D, off


@pytest.mark.parametrize("seed", range(30))
def test_variants_bruteforce_tiny(seed):
    rng = np.random.default_rng(7000 + seed)
    B = int(rng.integers(1, 4))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 8)), vocab=int(rng.integers(2, 5)))
    reqs = [tr.tokens[int(a):int(b)].tolist() for a, b in zip(tr.req_tok_off[:-1], tr.req_tok_off[1:])]
    blocks = bf_requests(reqs, B)
    ids, D, off = _setup(tr, B)
    kind = int(rng.integers(0, 3))
    f_lin, f_attn = int(rng.integers(0, 1000)), int(rng.integers(0, 1000))
    caps = list(range(1, D + 2))
    for order, res in VARIANTS:
        want = bf_sd(blocks, order, res)
        assert oracle.sd_variant(ids, D, off, order, res).tolist() == want, (order, res)
        assert oracle.sd_variant(ids, D, off, order, res, mattson=True).tolist() == want, (order, res)
        hits, saved = oracle.lru_curves_variant(ids, off, B, caps, order, res, kind, f_lin, f_attn)
        for C, h, s in zip(caps, hits, saved):
            assert (h, s) == bf_lru(blocks, B, C, order, res, kind, f_lin, f_attn), (order, res, C)


def test_root_first_per_block_is_the_hot_path():
    tr = tracegen.make(0).head(400)
    ids, D, off = _setup(tr, 16)
    sd = oracle.sd_fenwick(oracle.reuse(ids, D)[0])
    assert np.array_equal(oracle.sd_variant(ids, D, off, oracle.ROOT_FIRST, oracle.RES_BLOCK), sd)
    caps = [1, 10, 100, 1000, 10_000]
    h0, s0, _ = oracle.lru_curves(ids, off, 16, caps)
    assert oracle.lru_curves_variant(ids, off, 16, caps, oracle.ROOT_FIRST, oracle.RES_BLOCK) == (h0, s0)


@pytest.mark.parametrize("order,res", VARIANTS)
def test_inclusion_running_max(order, res):
    """Mattson inclusion under every variant: block k of a request counts at
    capacity C iff the largest distance over its depths 0..k is <= C."""
    tr = tracegen.make(0).head(300)
    ids, D, off = _setup(tr, 16)
    sd = oracle.sd_variant(ids, D, off, order, res).astype(np.int64)
    sd[sd == NONE] = 1 << 40
    e = np.empty_like(sd)
    for r in range(len(off) - 1):
        a, b = int(off[r]), int(off[r + 1])
        if b > a:
            e[a:b] = np.maximum.accumulate(sd[a:b])
    caps = [1, 3, 17, 64, 300, 2000, 50_000]
    hits, _ = oracle.lru_curves_variant(ids, off, 16, caps, order, res, oracle.COST_UNIFORM)
    assert hits == [int((e <= C).sum()) for C in caps]


def test_growing_session_closed_forms():
    """One session whose requests each extend the previous one (B = 1; n_t
    blocks at request t).  Re-read blocks k < n_{t-1} of request t have:
      root-first, per block:    distance n_{t-1}   (the window holds the previous context)
      root-first, per request:  distance n_{t-1} - k (the root is the oldest)
      leaf-first, per block:    distance n_t        (new blocks are touched first)
      leaf-first, per request:  distance k + 1      (the root is the most recent)"""
    rng = np.random.default_rng(3)
    ctx, reqs = [], []
    for _ in range(10):
        ctx = ctx + [int(x) for x in rng.integers(0, 10_000, int(rng.integers(1, 9)))]
        reqs.append(list(ctx))
    tr = tracegen.from_lists(reqs)
    ids, D, off = _setup(tr, 1)
    n = np.diff(off).astype(int)
    want = {v: [] for v in VARIANTS}
    for t in range(len(n)):
        for k in range(n[t]):
            old = t > 0 and k < n[t - 1]
            want[(0, 0)].append(n[t - 1] if old else NONE)
            want[(0, 1)].append(n[t - 1] - k if old else NONE)
            want[(1, 0)].append(n[t] if old else NONE)
            want[(1, 1)].append(k + 1 if old else NONE)
    for v in VARIANTS:
        assert oracle.sd_variant(ids, D, off, *v).tolist() == want[v], v
    # hits under per-request residency with the root most recent: min(C, n_{t-1}) per request
    caps = list(range(1, int(n.max()) + 2))
    hits, _ = oracle.lru_curves_variant(ids, off, 1, caps, oracle.LEAF_FIRST, oracle.RES_REQUEST, oracle.COST_UNIFORM)
    assert hits == [sum(min(C, int(n[t - 1])) for t in range(1, len(n))) for C in caps]


def test_bad_variant_rejected():
    ids = np.zeros(1, dtype=np.uint32)
    off = np.array([0, 1], dtype=np.uint64)
    with pytest.raises(ValueError):
        oracle.sd_variant(ids, 1, off, 2, 0)
    with pytest.raises(ValueError):
        oracle.lru_curves_variant(ids, off, 1, [1], 0, 3)


@pytest.mark.parametrize("seed", range(10))
def test_root_first_residency_leaves_hits_unchanged(seed):
    """Root-first, whole-request residency counts the same hits as per-block
    lookups.  Either way a counted block's shallower blocks were all found
    resident, so touching them root-first only moved them to the front and
    evicted nothing: the block's residency when touched is its residency at
    arrival."""
    rng = np.random.default_rng(8800 + seed)
    B = int(rng.integers(1, 4))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(2, 9)), vocab=int(rng.integers(2, 5)))
    ids, D, off = _setup(tr, B)
    caps = list(range(1, D + 2))
    per_block = oracle.lru_curves_variant(ids, off, B, caps, oracle.ROOT_FIRST, oracle.RES_BLOCK)
    per_request = oracle.lru_curves_variant(ids, off, B, caps, oracle.ROOT_FIRST, oracle.RES_REQUEST)
    assert per_block == per_request
