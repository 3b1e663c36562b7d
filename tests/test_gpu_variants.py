"""Stack distances and curves under the semantics variants (Sec. 3.1: touch
order, whole-request residency) on the GPU against the oracle, through the
C ABI: distances element by element, hits and compute saved at every
capacity, bit-exact."""
import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu
NONE = 0xFFFFFFFF
VARIANTS = [(o, r) for o in (0, 1) for r in (0, 1)]


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_28870_gb300 as ptc
    ptc.lib()


def _gpu_arrays(tr, B):
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util
    tok, off, ts = gpu_util.to_gpu(tr)
    tok = tok[: tr.tokens.size] if tr.tokens.size else tok[:0]
    return ptc.pipeline(tok, off, ts, B, [1])


def _variant(out, order, res, method=None):
    import paper_2609_28870_gb300 as ptc
    return ptc.ptc_stack_distance_variant(out["prev"], out["req_blk_off"], order, res, method=method)


@pytest.mark.parametrize("seed", range(20))
def test_tiny_random_traces_all_variants(seed):
    import paper_2609_28870_gb300 as ptc
    rng = np.random.default_rng(4000 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 10)), max_turns=int(rng.integers(1, 8)),
                       vocab=int(rng.integers(2, 5)))
    out = _gpu_arrays(tr, B)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    off = oracle.block_offsets(tr.req_tok_off, B)
    caps = list(range(1, D + 2))
    kind = int(rng.integers(0, 3))
    for order, res in VARIANTS:
        d = _variant(out, order, res)
        want = oracle.sd_variant(ids, D, off, order, res)
        assert np.array_equal(ptc.u32(d), want), (order, res)
        for method in (ptc.PTC_SD_POINTS, ptc.PTC_SD_RUNS):  # both routes of per-request residency
            assert np.array_equal(ptc.u32(_variant(out, order, res, method)), want), (order, res, method)
        if ids.size == 0:
            continue
        cur = ptc.ptc_curves(d, out["req_blk_off"], B, caps, kind=kind, f_lin=17, f_attn=5)
        h, s = oracle.lru_curves_variant(ids, off, B, caps, order, res, kind, 17, 5)
        assert cur["hits"] == h and cur["saved"] == s, (order, res)


def test_root_first_per_block_is_stack_distance():
    import paper_2609_28870_gb300 as ptc
    tr = tracegen.make(0)
    out = _gpu_arrays(tr, 16)
    assert np.array_equal(ptc.u32(_variant(out, 0, 0)), ptc.u32(out["dist"]))


@pytest.mark.parametrize("order,res", VARIANTS)
def test_tiny_conversational_workload(order, res):
    import paper_2609_28870_gb300 as ptc
    tr = tracegen.make(0)
    out = _gpu_arrays(tr, 16)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    off = oracle.block_offsets(tr.req_tok_off, 16)
    d = _variant(out, order, res)
    want = oracle.sd_variant(ids, D, off, order, res)
    assert np.array_equal(ptc.u32(d), want)
    for method in (ptc.PTC_SD_POINTS, ptc.PTC_SD_RUNS):
        assert np.array_equal(ptc.u32(_variant(out, order, res, method)), want), method
    caps = tracegen.workload_grid(0, D)
    cur = ptc.ptc_curves(d, out["req_blk_off"], 16, caps)
    h, s = oracle.lru_curves_variant(ids, off, 16, caps, order, res)
    assert cur["hits"] == h and cur["saved"] == s


def test_chat_workload_full_size_all_variants():
    """The chat workload (~9.6M accesses): distances of every variant
    element by element; hits at every grid point by inclusion from the
    oracle's distances; direct LRU at two capacities per variant."""
    import paper_2609_28870_gb300 as ptc
    tr = tracegen.make(1)
    out = _gpu_arrays(tr, 16)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    off = oracle.block_offsets(tr.req_tok_off, 16)
    caps = tracegen.workload_grid(1, D)
    lens = np.diff(off).astype(np.int64)
    starts = np.repeat(off[:-1].astype(np.int64), lens)
    for order, res in VARIANTS:
        d = _variant(out, order, res)
        sd = oracle.sd_variant(ids, D, off, order, res)
        assert np.array_equal(ptc.u32(d), sd), (order, res)
        cur = ptc.ptc_curves(d, out["req_blk_off"], 16, caps)
        # running max over depth within each request, then inclusion
        x = sd.astype(np.int64)
        x[sd == NONE] = 1 << 40
        e = x.copy()
        for r in np.flatnonzero(lens > 1):  # per request (the trace has ~17K)
            a, b = int(off[r]), int(off[r + 1])
            e[a:b] = np.maximum.accumulate(x[a:b])
        assert cur["hits"] == [int((e <= c).sum()) for c in caps], (order, res)
        pick = [len(caps) // 4, 3 * len(caps) // 4]
        h, s = oracle.lru_curves_variant(ids, off, 16, caps[pick], order, res)
        assert [cur["hits"][p] for p in pick] == h and [cur["saved"][p] for p in pick] == s
    assert starts.size == ids.size


def test_edge_cases_and_errors():
    import torch
    import paper_2609_28870_gb300 as ptc
    # one request, one block; requests without full blocks in between
    tr = tracegen.from_lists([[5, 6], [], [5], [5, 6, 7, 8], [7, 7, 7, 7]])
    out = _gpu_arrays(tr, 2)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 2)
    off = oracle.block_offsets(tr.req_tok_off, 2)
    for order, res in VARIANTS:
        assert np.array_equal(ptc.u32(_variant(out, order, res)), oracle.sd_variant(ids, D, off, order, res))
    # an empty trace
    e = ptc.ptc_stack_distance_variant(torch.zeros(0, dtype=torch.int32, device="cuda"),
                                       torch.zeros(3, dtype=torch.int64, device="cuda"), 1, 1)
    assert e.numel() == 0
    # bad variant values, a forward prev, malformed offsets
    with pytest.raises(ptc.PtcError):
        ptc.ptc_stack_distance_variant(out["prev"], out["req_blk_off"], 2, 0)
    with pytest.raises(ptc.PtcError):
        ptc.ptc_stack_distance_variant(out["prev"], out["req_blk_off"], 0, 1, method=7)
    prev = out["prev"].clone()
    prev[0] = 2
    for order, res in [(1, 0), (0, 1), (1, 1)]:
        for method in (None, ptc.PTC_SD_POINTS, ptc.PTC_SD_RUNS):
            with pytest.raises(ptc.PtcError) as ex:
                ptc.ptc_stack_distance_variant(prev, out["req_blk_off"], order, res, method=method)
            assert ex.value.name == "PTC_ERR_INVALID_ARG"
    bad_off = out["req_blk_off"].clone()
    bad_off[-1] = bad_off[-1] + 5
    for order, res in [(1, 0), (0, 1), (1, 1)]:
        with pytest.raises(ptc.PtcError):
            ptc.ptc_stack_distance_variant(out["prev"], bad_off, order, res)
    # still usable
    assert np.array_equal(ptc.u32(_variant(out, 1, 1)), oracle.sd_variant(ids, D, off, 1, 1))
