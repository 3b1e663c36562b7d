"""Parity at the full sizes of the agentic (2.08B tokens, 130M accesses),
agentic-at-other-block-sizes and mixed 24-hour (10.0B tokens, 624M accesses)
workloads, in the launch configuration the bench times (ptc_pipeline, one C
call, session labels given, caller arrays for every intermediate).

The agentic trace at B = 16 is compared with the oracle run live, element by
element.  The other block sizes and the mixed trace are compared with the
oracle's stored results (tests/golden/big_configs.json, written by
tests/golden/make_big_goldens.py, which runs the oracle alone): SHA-256 of
every per-access array (ids, prev, next, stack distances), N and D, hits and
128-bit compute saved at every grid point, the total cost, and the direct
per-capacity LRU simulation at several grid points.  On top of that, what
holds at any size is checked from the GPU's own arrays:
  * sampled accesses against the definitions themselves (same id iff same
    prefix, by token comparison; prev is the last earlier access with the id;
    the stack distance is one plus the distinct ids strictly between);
  * the identities of the method (next[prev[i]] = i, D first accesses,
    Mattson inclusion for every grid point, the cost totals in closed form)."""
import hashlib
import json
import os

import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu
NONE = 0xFFFFFFFF


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "big_configs.json")


def _sha(a):
    h = hashlib.sha256()
    mv = memoryview(np.ascontiguousarray(a)).cast("B")
    for i in range(0, len(mv), 1 << 28):
        h.update(mv[i:i + (1 << 28)])
    return h.hexdigest()


def _golden(key):
    if not os.path.exists(GOLDEN):
        pytest.fail("tests/golden/big_configs.json is missing: run tests/golden/make_big_goldens.py")
    with open(GOLDEN) as f:
        g = json.load(f)
    if key not in g:
        pytest.fail(f"{key} is missing from tests/golden/big_configs.json")
    return g[key]


def _against_golden(g, gold, tr, caps):
    """Every output of the GPU run against the oracle's stored results."""
    assert _sha(tr.tokens) == gold["tokens_sha256"] and _sha(tr.req_tok_off) == gold["req_tok_off_sha256"]
    assert g["n_access"] == gold["N"] and g["n_distinct"] == gold["D"]
    for k in ("ids", "prev", "next", "dist"):
        assert _sha(g[k]) == gold[k + "_sha256"], k
    assert [int(c) for c in caps] == gold["caps"]
    assert g["hits"] == gold["hits"]
    assert [str(x) for x in g["saved"]] == gold["saved"]
    assert str(g["total_cost"]) == gold["total_cost"]
    d = gold["direct"]
    for idx, h, s in zip(d["index"], d["hits"], d["saved"]):
        assert g["hits"][idx] == h and str(g["saved"][idx]) == s


def _sessions(tr):
    import torch
    return torch.from_numpy(np.ascontiguousarray(tr.req_session, dtype=np.uint32).view(np.int32)).cuda()


def _pipeline(tok, off, ts, n_tok, n_req, B, caps, ses=None, n_session=0):
    """ptc_pipeline with caller arrays for every intermediate; numpy results."""
    import torch
    import paper_2609_28870_gb300 as ptc
    nmax = max(n_tok // B, 1)
    outs = {k: torch.empty(nmax, dtype=torch.int32, device="cuda") for k in ("ids", "prev", "next", "dist")}
    outs["keys"] = torch.empty(2 * nmax, dtype=torch.int64, device="cuda")
    outs["req_blk_off"] = torch.empty(n_req + 1, dtype=torch.int64, device="cuda")
    res = ptc.ptc_pipeline(tok, off, ts, B, caps, outputs=outs, req_session=ses, n_session=n_session)
    n = res["n_access"]
    for k in ("ids", "prev", "next", "dist"):
        res[k] = outs[k][:n].cpu().numpy().view(np.uint32)
    res["keys"] = outs["keys"].view(torch.int64)[: 2 * n].cpu().numpy().view(np.uint64).reshape(-1, 2)
    res["req_blk_off"] = outs["req_blk_off"].cpu().numpy().view(np.uint64)
    del outs
    torch.cuda.empty_cache()
    return res


def _to_gpu(tr):
    import torch
    import paper_2609_28870_gb300 as ptc
    return (ptc.to_device_u32(tr.tokens), ptc.to_device_u64(tr.req_tok_off),
            torch.from_numpy(np.ascontiguousarray(tr.req_ts_us)).cuda())


def _cost(k, B):
    """Per-block cost of the measured model (u64, exact: below 2^63 here)."""
    k = k.astype(np.uint64)
    return (np.uint64(B * oracle.F_LIN) + np.uint64(oracle.F_ATTN) *
            (np.uint64(B * B) * k + np.uint64(B * (B + 1) // 2)))


def _exact_sum(v):
    """Exact Python integer sum of a uint64 array (split into 32-bit halves)."""
    lo = (v & np.uint64(0xFFFFFFFF)).sum(dtype=np.uint64)
    hi = (v >> np.uint64(32)).sum(dtype=np.uint64)
    return int(lo) + (int(hi) << 32)


def _identities(g, B, caps, tr):
    """What holds at any size: cold counts, next/prev inverse, inclusion
    (hits and saved from the stack distances), monotonicity, cost total."""
    N, D = g["n_access"], g["n_distinct"]
    prev, nxt, sd, ids = g["prev"], g["next"], g["dist"], g["ids"]
    off = oracle.block_offsets(tr.req_tok_off, B)
    assert np.array_equal(g["req_blk_off"], off) and N == int(off[-1])
    cold = prev == NONE
    assert int(cold.sum()) == D and int((nxt == NONE).sum()) == D
    nc = np.flatnonzero(~cold)
    assert np.all(nxt[prev[nc]] == nc)
    assert np.array_equal(sd == NONE, cold)
    # first occurrences are numbered 0, 1, 2, ... in access order
    assert np.array_equal(ids[cold], np.arange(D, dtype=np.uint32))
    assert np.all(ids[nc] == ids[prev[nc]])
    # block index within the request of every access, and its cost
    k = np.arange(N, dtype=np.uint64) - np.repeat(off[:-1], np.diff(off).astype(np.int64))
    cost = _cost(k, B)
    del k
    assert g["total_cost"] == _exact_sum(cost)
    # Mattson inclusion at every grid point: an access hits at c iff sd <= c.
    # Bin each access at the first grid point it hits at; costs go in as
    # three 21-bit limbs so every float bin sum stays exact (below 2^53).
    capa = np.asarray(caps, dtype=np.uint64)
    gidx = np.searchsorted(capa, sd.astype(np.uint64), side="left")  # cold (NONE) lands past the end
    G = capa.size
    hits_bins = np.bincount(gidx, minlength=G + 1)[:G]
    limbs = [np.bincount(gidx, weights=((cost >> np.uint64(21 * j)) & np.uint64((1 << 21) - 1)).astype(np.float64),
                         minlength=G + 1)[:G] for j in range(3)]
    run_h, run_s = 0, 0
    for gi in range(G):
        run_h += int(hits_bins[gi])
        run_s += sum(int(limbs[j][gi]) << (21 * j) for j in range(3))
        assert g["hits"][gi] == run_h and g["saved"][gi] == run_s
    return off


def _sampled_definitions(g, tr, B, off, rng, n_samples=300, window_cap=2_000_000):
    """Sampled accesses against the definitions (token comparison, window scans)."""
    ids, prev, sd = g["ids"], g["prev"], g["dist"]
    N = g["n_access"]
    tok, toff = tr.tokens, tr.req_tok_off

    def req_of(i):
        return int(np.searchsorted(off, np.uint64(i), side="right")) - 1

    def prefix(i):
        r = req_of(i)
        kk = i - int(off[r])
        return tok[int(toff[r]): int(toff[r]) + B * (kk + 1)]

    checked = 0
    for i in rng.choice(N, n_samples, replace=False):
        i = int(i)
        p = int(prev[i])
        if p != NONE:
            assert np.array_equal(prefix(i), prefix(p))  # same id iff same prefix
            if i - p <= window_cap:
                win = ids[p + 1: i]
                assert not np.any(win == ids[i])  # no use of the id in between
                assert int(sd[i]) == 1 + np.unique(win).size
                checked += 1
        # the key of the block is the prefix hash of the oracle
        r = req_of(i)
        one = np.array([0, B * (i - int(off[r]) + 1)], dtype=np.uint64)
        kh = oracle.prefix_hash(prefix(i), one, B, 0)
        assert np.array_equal(g["keys"][i], kh[-1])
    assert checked > n_samples // 10


@pytest.fixture(scope="module")
def agentic():
    tr = tracegen.make(2)
    dev = _to_gpu(tr)
    ses = _sessions(tr)
    # D at B = 16 sets the token-denominated grid of the other block sizes
    # (the value itself is pinned by test_agentic_full_size)
    d16 = _pipeline(*dev, tr.tokens.size, tr.n_req, 16, [1])["n_distinct"]
    return tr, dev, ses, d16


def test_agentic_full_size(agentic):
    """Agentic workload, B = 16, at full size, with and without session
    labels: every per-access array against the oracle run here, the curves by
    direct LRU simulation at two capacities and by inclusion at all 64."""
    tr, (tok, off_d, ts), ses, d16 = agentic
    B = 16
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    assert D == d16
    caps = tracegen.workload_grid(2, D)
    g = _pipeline(tok, off_d, ts, tr.tokens.size, tr.n_req, B, caps, ses, tr.n_sessions)
    assert g["n_distinct"] == D and np.array_equal(g["ids"], ids)
    prev, nxt = oracle.reuse(ids, D)
    assert np.array_equal(g["prev"], prev) and np.array_equal(g["next"], nxt)
    sd = oracle.sd_fenwick(prev)
    assert np.array_equal(g["dist"], sd)
    off = _identities(g, B, caps, tr)
    pick = [len(caps) // 4, 3 * len(caps) // 4]
    h, s, t = oracle.lru_curves(ids, off, B, caps[pick])
    assert [g["hits"][p] for p in pick] == h and [g["saved"][p] for p in pick] == s
    assert g["total_cost"] == t
    _sampled_definitions(g, tr, B, off, np.random.default_rng(2), n_samples=100)
    # without sessions (every key through the table): the same results
    g2 = _pipeline(tok, off_d, ts, tr.tokens.size, tr.n_req, B, caps)
    for k in ("ids", "prev", "next", "dist"):
        assert np.array_equal(g2[k], g[k]), k
    assert g2["hits"] == g["hits"] and g2["saved"] == g["saved"]


@pytest.mark.parametrize("B", [16, 32, 64, 256])
def test_agentic_block_sizes_against_golden(agentic, B):
    """The agentic trace re-blocked at B = 16, 32, 64, 256 (the block-size
    study) with the token-denominated capacity grid, against the oracle's
    stored results: every per-access array, the curves at all grid points and
    the direct LRU simulation at four of them."""
    tr, (tok, off_d, ts), ses, d16 = agentic
    gold = _golden(f"agentic_B{B}")
    # capacities in tokens: 16 x a mixed-style grid over D at B = 16, as blocks of B
    base = tracegen.capacity_grid(max(1, round(0.001 * d16)), d16, 128).astype(np.uint64)
    caps = np.unique(np.maximum(np.uint64(1), (np.uint64(16) * base) // np.uint64(B)))
    g = _pipeline(tok, off_d, ts, tr.tokens.size, tr.n_req, B, caps, ses, tr.n_sessions)
    _against_golden(g, gold, tr, caps)
    _identities(g, B, caps, tr)


def test_mixed_full_size():
    """Mixed 24-hour workload (10.0B tokens, 624M accesses) at full size,
    B = 16, 128-point grid, with session labels as the bench runs it: every
    output against the oracle's stored results; sampled accesses against the
    definitions; the identities over all accesses."""
    tr = tracegen.make(3)
    gold = _golden("mixed_B16")
    tok, off_d, ts = _to_gpu(tr)
    ses = _sessions(tr)
    B = 16
    caps = tracegen.workload_grid(3, gold["D"])
    g = _pipeline(tok, off_d, ts, tr.tokens.size, tr.n_req, B, caps, ses, tr.n_sessions)
    del tok, off_d, ts, ses
    _against_golden(g, gold, tr, caps)
    off = _identities(g, B, caps, tr)
    _sampled_definitions(g, tr, B, off, np.random.default_rng(3), n_samples=200)
