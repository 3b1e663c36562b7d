"""GPU path vs the CPU oracle, element by element, through the C-ABI.

Everything here is integer work, so the bar is bit-exact: block keys,
request block offsets, ids, distinct count, prev / next, stack distances,
per-capacity hits and the 128-bit compute-saved sums."""
import json
import os

import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_28870_gb300 as ptc
    ptc.lib()


def _g():
    from tests import gpu_util
    return gpu_util


def test_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "worked_example.json")))
    tr = tracegen.from_lists(g["requests"])
    cm = g["cost_model"]
    res = _g().gpu_run(tr, g["block_size"], g["capacities"], cm["kind"], 0, cm["f_lin"], cm["f_attn"])
    none = lambda v: [0xFFFFFFFF if x is None else x for x in v]
    assert res["ids"].tolist() == g["ids"]
    assert res["prev"].tolist() == none(g["prev"])
    assert res["next"].tolist() == none(g["next"])
    assert res["dist"].tolist() == none(g["sd"])
    assert res["hits"] == g["hits"] and res["saved"] == g["saved"] and res["total_cost"] == g["total_cost"]


@pytest.mark.parametrize("seed", range(30))
def test_tiny_random_traces(seed):
    rng = np.random.default_rng(5000 + seed)
    B = int(rng.choice([1, 2, 3, 4, 5, 7, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 12)), max_turns=6, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 40)))
    kind = int(rng.integers(0, 3))
    o0 = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    caps = list(range(1, o0[1] + 2)) or [1]
    gu = _g()
    g = gu.gpu_run(tr, B, caps, kind, seed=seed)
    o = gu.oracle_run(tr, B, caps, kind)
    gu.assert_same(g, o)
    assert np.array_equal(g["keys"], oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, seed))


@pytest.mark.parametrize("B", [16, 32, 64, 256, 48, 500])
def test_agentic_block_sizes(B):
    """The agentic generator at reduced scale, rehashed at several block sizes
    (including ones that are not a multiple of 16)."""
    tr = tracegen.make(2, sessions=12)
    gu = _g()
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    caps = tracegen.capacity_grid(1, D, 128)
    g = gu.gpu_run(tr, B, caps, seed=B)
    o = gu.oracle_run(tr, B, caps)
    gu.assert_same(g, o)
    assert np.array_equal(g["keys"][:2000], oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, B)[:2000])


def test_tiny_conversational_workload_full():
    """The tiny conversational workload (seed 0) end to end, 16-point grid."""
    tr = tracegen.make(0)
    gu = _g()
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(0, D)
    g = gu.gpu_run(tr, 16, caps)
    o = gu.oracle_run(tr, 16, caps)
    gu.assert_same(g, o)
    for kind in (0, 2):
        g2 = gu.gpu_run(tr, 16, caps, kind)
        h, s, t = oracle.lru_curves(o["ids"], o["req_blk_off"], 16, caps, kind)
        assert g2["hits"] == h and g2["saved"] == s and g2["total_cost"] == t


def test_chat_workload_full_size():
    """The conversational chat workload at full size (~154M tokens, ~9.6M
    accesses), as the bench runs it: every per-access array bit-exact against
    the oracle; the curves exact at four sampled capacities by direct LRU
    simulation and at every grid point by the oracle's own stack distances."""
    tr = tracegen.make(1)
    gu = _g()
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(1, D)
    g = gu.gpu_run(tr, 16, caps)
    off = oracle.block_offsets(tr.req_tok_off, 16)
    assert np.array_equal(g["req_blk_off"], off)
    assert g["n_distinct"] == D and np.array_equal(g["ids"], ids)
    prev, nxt = oracle.reuse(ids, D)
    assert np.array_equal(g["prev"], prev) and np.array_equal(g["next"], nxt)
    sd = oracle.sd_fenwick(prev)
    assert np.array_equal(g["dist"], sd)
    pick = [0, len(caps) // 3, 2 * len(caps) // 3, len(caps) - 1]
    h, s, t = oracle.lru_curves(ids, off, 16, caps[pick])
    assert [g["hits"][p] for p in pick] == h
    assert [g["saved"][p] for p in pick] == s
    assert g["total_cost"] == t
    # every grid point via Mattson inclusion on the oracle's distances
    finite = sd != oracle.NONE
    exp = [int((finite & (sd <= c)).sum()) for c in caps]
    assert g["hits"] == exp
    sample = np.random.default_rng(0).choice(g["keys"].shape[0], 2000, replace=False)
    small = tr.head(300)
    keys_o = oracle.prefix_hash(small.tokens, small.req_tok_off, 16, 0)
    assert np.array_equal(g["keys"][: keys_o.shape[0]], keys_o)
    assert sample.size == 2000


def test_edge_cases():
    gu = _g()
    cases = [
        [[1, 2, 3]],                          # one request, one block at B=2, tail dropped
        [[5] * 64] * 5,                       # identical requests
        [[], [1], [], [1, 2, 3, 4], []],      # empty and short requests
        [[0xFFFFFFFF, 0, 0xFFFFFFFF, 0]] * 3,  # extreme token values
        [list(range(40)), list(range(40))[::-1], list(range(40))],
    ]
    for reqs in cases:
        tr = tracegen.from_lists(reqs)
        for B in (1, 2, 3, 16):
            ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
            if ids.size == 0:
                continue
            caps = list(range(1, D + 2))
            gu.assert_same(gu.gpu_run(tr, B, caps), gu.oracle_run(tr, B, caps))


def test_empty_trace_and_no_blocks():
    import paper_2609_28870_gb300 as ptc
    import torch
    gu = _g()
    tr = tracegen.from_lists([[1, 2], [3]])
    tok, off, ts = gu.to_gpu(tr)
    keys, blk_off, n = ptc.ptc_hash_blocks(tok[:3], off, ts, 16, 0)
    assert n == 0 and ptc.u64(blk_off).tolist() == [0, 0, 0]
    e = tracegen.from_lists([])
    off0 = ptc.to_device_u64(e.req_tok_off)
    keys, blk_off, n = ptc.ptc_hash_blocks(torch.zeros(1, dtype=torch.int32, device="cuda"), off0, None, 16, 0)
    assert n == 0
    ids, d = ptc.ptc_assign_ids(keys)
    assert d == 0 and ids.numel() == 0
    cur = ptc.ptc_curves(torch.zeros(0, dtype=torch.int32, device="cuda"), blk_off, 16, [1, 2])
    assert cur["hits"] == [0, 0] and cur["total_cost"] == 0


def test_unaligned_token_pointer():
    """A token buffer that starts 4 bytes past a 16-byte boundary."""
    import paper_2609_28870_gb300 as ptc
    tr = tracegen.tiny(3, n_sessions=6, vocab=4, max_seg=30)
    gu = _g()
    big = np.concatenate([np.zeros(1, np.uint32), tr.tokens])
    tok = ptc.to_device_u32(big)[1:]
    off = ptc.to_device_u64(tr.req_tok_off)
    keys, blk_off, n = ptc.ptc_hash_blocks(tok, off, None, 3, 11)
    assert np.array_equal(ptc.u64(keys).reshape(-1, 2), oracle.prefix_hash(tr.tokens, tr.req_tok_off, 3, 11))


def test_error_statuses():
    import paper_2609_28870_gb300 as ptc
    import torch
    gu = _g()
    tr = tracegen.tiny(1, n_sessions=4)
    tok, off, ts = gu.to_gpu(tr)
    bad_ts = ts.flip(0).contiguous()
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_hash_blocks(tok, off, bad_ts, 2, 0)
    assert e.value.name == "PTC_ERR_UNSORTED"
    bad_off = off.clone()
    bad_off[-1] = tr.tokens.size + 100
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_hash_blocks(tok, bad_off, None, 2, 0)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_hash_blocks(tok, off, ts, 1, 0, keys_cap=1)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    keys, blk_off, n = ptc.ptc_hash_blocks(tok, off, ts, 1, 0)
    ids, d = ptc.ptc_assign_ids(keys)
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_reuse_indices(ids, max(1, d - 1))
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    small = torch.empty(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(ptc.PtcError) as e:
        ptc.lib()  # the raw call with an undersized workspace
        rc = ptc.lib().ptc_stack_distance(ids.data_ptr(), ids.numel(), ids.data_ptr(), small.data_ptr(), 256,
                                          torch.cuda.current_stream().cuda_stream)
        ptc._check("ptc_stack_distance", rc)
    assert e.value.name == "PTC_ERR_WORKSPACE"
    prev = torch.arange(ids.numel(), dtype=torch.int32, device="cuda")  # prev[i] = i is malformed
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_stack_distance(prev)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_curves(ptc.ptc_stack_distance(ptc.ptc_reuse_indices(ids, d)[0]), blk_off, 1, [3, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"


def test_verify_ids_exact_and_detects_merge():
    import paper_2609_28870_gb300 as ptc
    gu = _g()
    tr = tracegen.make(0, max_requests=200)
    tok, off, ts = gu.to_gpu(tr)
    keys, blk_off, n = ptc.ptc_hash_blocks(tok, off, ts, 16, 0)
    ids, d = ptc.ptc_assign_ids(keys)
    ptc.ptc_verify_ids(tok, off, blk_off, 16, ids, d)
    # merge two different blocks under one id: the exact check must object
    bad = ids.clone()
    a = int(np.nonzero(ptc.u32(ids) == 1)[0][0])
    bad[a] = 0
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_verify_ids(tok, off, blk_off, 16, bad, d)
    assert e.value.name == "PTC_ERR_HASH_COLLISION"


def test_deterministic_repeat():
    tr = tracegen.make(0, max_requests=600)
    gu = _g()
    caps = tracegen.capacity_grid(16, 50000, 32)
    a = gu.gpu_run(tr, 16, caps)
    b = gu.gpu_run(tr, 16, caps)
    for k in ("keys", "ids", "prev", "next", "dist"):
        assert np.array_equal(a[k], b[k])
    assert a["hits"] == b["hits"] and a["saved"] == b["saved"]


def test_all_distinct_blocks_take_the_full_table():
    """One long request: every block is distinct (different prefix lengths),
    so the first, smaller hash table overflows and the call redoes the stage
    with the full one."""
    rng = np.random.default_rng(9)
    tr = tracegen.from_lists([rng.integers(0, 2**32, 60000, dtype=np.uint64).tolist()])
    gu = _g()
    caps = [1, 2, 100]
    g = gu.gpu_run(tr, 1, caps)
    o = gu.oracle_run(tr, 1, caps)
    gu.assert_same(g, o)
    assert g["n_distinct"] == 60000


def test_long_runs_and_run_breaks():
    """Stack distances over long copied runs (a run's accesses share one
    distance) with runs broken by truncation, interleaving and cold blocks."""
    reqs, ctx = [], []
    rng = np.random.default_rng(4)
    for t in range(30):
        ctx = ctx + rng.integers(0, 1000, int(rng.integers(40, 400))).tolist()
        if t % 7 == 6:
            ctx = ctx[:30] + ctx[200:]  # truncation breaks the run
        reqs.append(list(ctx))
        reqs.append(rng.integers(0, 1000, 50).tolist())  # an unrelated request in between
    tr = tracegen.from_lists(reqs)
    gu = _g()
    for B in (1, 4, 16):
        ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
        caps = tracegen.capacity_grid(1, D + 1, 40)
        gu.assert_same(gu.gpu_run(tr, B, caps), gu.oracle_run(tr, B, caps))


@pytest.mark.parametrize("vocab", [2**32 - 1, 2**27 + 5])
def test_full_range_token_values(vocab):
    """Tokens up to 2^32 - 1 at B = 16 with 16-byte-aligned tokens: blocks
    whose tokens all fit 27 bits and blocks that need the three-limb
    products sit in the same warps; keys, ids and curves bit-exact."""
    rng = np.random.default_rng(vocab & 0xFFFF)
    reqs = []
    for s in range(40):
        base = [int(x) for x in rng.integers(0, vocab if s % 3 else 151936, size=int(rng.integers(16, 400)))]
        reqs.append(base)
        reqs.append(base + [int(x) for x in rng.integers(0, vocab, size=int(rng.integers(0, 200)))])
    tr = tracegen.from_lists(reqs)
    gu = _g()
    _, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = list(range(1, D + 2, max(1, D // 40)))
    g = gu.gpu_run(tr, 16, caps, seed=77)
    gu.assert_same(g, gu.oracle_run(tr, 16, caps))
    assert np.array_equal(g["keys"], oracle.prefix_hash(tr.tokens, tr.req_tok_off, 16, 77))
