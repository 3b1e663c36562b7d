"""ptc_pipeline (the five stages in one C call) against the CPU oracle,
bit-exact, with and without caller-supplied output arrays."""
import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_28870_gb300 as ptc
    ptc.lib()


def _run(tr, B, caps, kind=oracle.COST_MEASURED, seed=0, with_outputs=True):
    import torch
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util as gu
    tok, off, ts = gu.to_gpu(tr)
    tok = tok[: tr.tokens.size]
    nmax = max(tr.tokens.size // B, 1)
    outs = None
    if with_outputs:
        outs = {k: torch.empty(nmax, dtype=torch.int32, device="cuda") for k in ("ids", "prev", "next", "dist")}
        outs["keys"] = torch.empty(2 * nmax, dtype=torch.int64, device="cuda")
        outs["req_blk_off"] = torch.empty(tr.n_req + 1, dtype=torch.int64, device="cuda")
    res = ptc.ptc_pipeline(tok, off, ts, B, caps, kind=kind, seed=seed, outputs=outs)
    if with_outputs:
        n = res["n_access"]
        for k in ("ids", "prev", "next", "dist"):
            res[k] = ptc.u32(outs[k])[:n]
        res["keys"] = ptc.u64(outs["keys"]).reshape(-1, 2)[:n]
        res["req_blk_off"] = ptc.u64(outs["req_blk_off"])
    return res


@pytest.mark.parametrize("seed", range(8))
def test_pipeline_tiny_random(seed):
    from tests import gpu_util as gu
    rng = np.random.default_rng(9000 + seed)
    B = int(rng.choice([1, 2, 3, 5, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 12)), max_turns=6, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 40)))
    kind = int(rng.integers(0, 3))
    _, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    caps = list(range(1, D + 2))
    g = _run(tr, B, caps, kind, seed)
    o = gu.oracle_run(tr, B, caps, kind)
    gu.assert_same(g, o)
    assert np.array_equal(g["keys"], oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, seed))
    # without caller arrays the keys skip their carry pass (stage a2 adds it)
    bare = _run(tr, B, caps, kind, seed, with_outputs=False)
    for k in ("n_access", "n_distinct", "hits", "saved", "total_cost"):
        assert bare[k] == o[k]


@pytest.mark.parametrize("B", [1, 5, 16])
def test_pipeline_without_outputs_across_hash_tiles(B):
    """Requests of thousands of blocks, so most keys take a carry from an
    earlier tile; the pipeline without caller arrays adds it in stage a2."""
    from tests import gpu_util as gu
    rng = np.random.default_rng(400 + B)
    base = list(rng.integers(0, 6, size=3000 * B))
    reqs = [base[: 1700 * B + 3], base[: 2600 * B], list(rng.integers(0, 6, size=900 * B)), base[: 3000 * B - 1],
            base[: 40 * B]]
    tr = tracegen.from_lists(reqs)
    _, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    caps = [1, 7, 64, 500, D + 1]
    o = gu.oracle_run(tr, B, caps)
    for with_outputs in (True, False):
        g = _run(tr, B, caps, with_outputs=with_outputs)
        for k in ("n_access", "n_distinct", "hits", "saved", "total_cost"):
            assert g[k] == o[k], (k, with_outputs)


def test_pipeline_conversational_matches_oracle_and_separate_calls():
    from tests import gpu_util as gu
    tr = tracegen.make(0)
    _, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(0, D)
    g = _run(tr, 16, caps)
    gu.assert_same(g, gu.oracle_run(tr, 16, caps))
    bare = _run(tr, 16, caps, with_outputs=False)
    for k in ("n_access", "n_distinct", "hits", "saved", "total_cost"):
        assert bare[k] == g[k]
    sep = gu.gpu_run(tr, 16, caps)
    assert sep["hits"] == g["hits"] and sep["saved"] == g["saved"]


def test_pipeline_degenerate_traces():
    import torch
    import paper_2609_28870_gb300 as ptc
    # requests shorter than a block: no accesses at all
    tr = tracegen.from_lists([[1, 2], [3]])
    r = _run(tr, 16, [1, 2])
    assert r["n_access"] == 0 and r["n_distinct"] == 0 and r["hits"] == [0, 0] and r["total_cost"] == 0
    assert r["req_blk_off"].tolist() == [0, 0, 0]
    # no requests
    e = tracegen.from_lists([])
    off0 = ptc.to_device_u64(e.req_tok_off)
    r = ptc.ptc_pipeline(torch.zeros(0, dtype=torch.int32, device="cuda"), off0, None, 16, [4])
    assert r["n_access"] == 0 and r["hits"] == [0] and r["saved"] == [0]
    # one request of one block
    tr = tracegen.from_lists([[7] * 16])
    r = _run(tr, 16, [1])
    assert r["n_access"] == 1 and r["n_distinct"] == 1 and r["hits"] == [0]
    assert r["dist"].tolist() == [0xFFFFFFFF]


def test_pipeline_rejects_bad_arguments():
    import ctypes
    import torch
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util as gu
    tr = tracegen.from_lists([[1] * 32])
    tok, off, ts = gu.to_gpu(tr)
    for B in (0, 513):
        with pytest.raises(ptc.PtcError) as ei:
            ptc.ptc_pipeline(tok[:32], off, ts, B, [1])
        assert ei.value.name == "PTC_ERR_INVALID_ARG"
    # a workspace below ptc_pipeline_workspace_bytes, through the C call itself
    L = ptc.lib()
    small = torch.empty(256, dtype=torch.uint8, device="cuda")
    n, d = ctypes.c_uint64(7), ctypes.c_uint64(7)
    hits, saved, total = np.zeros(1, np.uint64), np.zeros(2, np.uint64), ptc.U128()
    caps = np.array([1], np.uint64)
    cm = ptc.CostModel(ptc.F_LIN, ptc.F_ATTN, ptc.PTC_COST_MEASURED)
    rc = L.ptc_pipeline(tok.data_ptr(), 32, off.data_ptr(), ts.data_ptr(), None, 0, 1, 16, 0, ctypes.byref(cm),
                        caps.ctypes.data, 1, None, None, None, None, None, None, ctypes.byref(n), ctypes.byref(d),
                        hits.ctypes.data, saved.ctypes.data, ctypes.byref(total), small.data_ptr(), 256,
                        torch.cuda.current_stream().cuda_stream)
    assert ptc.STATUS[rc] == "PTC_ERR_WORKSPACE"


def test_pipeline_reports_stage_a1_errors():
    """Stage a1 does not wait for its own status inside ptc_pipeline: its
    error word reaches the caller through stage a2's wait, and stage a2 must
    stay inside the keys buffer whatever N stage a1 left."""
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util as gu
    tr = tracegen.tiny(1, n_sessions=4)
    tok, off, ts = gu.to_gpu(tr)
    bad_off = off.clone()
    bad_off[-1] = tr.tokens.size + 100  # the last request runs past the tokens
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_pipeline(tok, bad_off, ts, 2, [1, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    bad_ts = ts.flip(0).contiguous()
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_pipeline(tok, off, bad_ts, 2, [1, 2])
    assert e.value.name == "PTC_ERR_UNSORTED"
    bad_off = off.clone()
    bad_off[1] = bad_off[2] + 5  # offsets that go backwards
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_pipeline(tok, bad_off, ts, 2, [1, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    # and a good call afterwards still matches the oracle (nothing stale in the slots)
    gu.assert_same(_run(tr, 2, [1, 2]), gu.oracle_run(tr, 2, [1, 2]))


def test_pipeline_plan_runs_again_and_on_refilled_buffers():
    """PipelinePlan marshals ptc_pipeline's arguments once: repeated runs give
    the same curves, and refilling its device buffers with another trace of
    the same shape gives that trace's curves."""
    import numpy as np
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util as gu
    tr_a = tracegen.tiny(5, n_sessions=6, max_turns=4, vocab=5, max_seg=30)
    rng = np.random.default_rng(12)
    tr_b = tracegen.from_lists([list(rng.integers(0, 5, size=int(tr_a.req_tok_off[r + 1] - tr_a.req_tok_off[r])))
                                for r in range(tr_a.n_req)])
    assert tr_b.tokens.size == tr_a.tokens.size and np.array_equal(tr_b.req_tok_off, tr_a.req_tok_off)
    B = 3
    caps = [1, 2, 4, 8, 16, 1000]
    tok, off, ts = gu.to_gpu(tr_a)
    tok = tok[: tr_a.tokens.size]
    plan = ptc.PipelinePlan(tok, off, None, B, caps)
    keys = ("n_access", "n_distinct", "hits", "saved", "total_cost")
    first = plan.run().result()
    o = gu.oracle_run(tr_a, B, caps)
    assert {k: first[k] for k in keys} == {k: o[k] for k in keys}
    assert plan.run().result() == first
    tok.copy_(ptc.to_device_u32(tr_b.tokens))
    second = plan.run().result()
    o = gu.oracle_run(tr_b, B, caps)
    assert {k: second[k] for k in keys} == {k: o[k] for k in keys}


def test_pipeline_redoes_stage_a2_when_the_small_table_overflows():
    """ptc_pipeline does not wait for stage a2: its first attempt uses the
    small table (N/3 slots); when every block is distinct that table
    overflows, stage b's wait reports it, and the pipeline redoes a2 with the
    full table and b with the host's N and D."""
    from tests import gpu_util as gu
    rng = np.random.default_rng(77)
    reqs = [list(rng.integers(0, 2**31, size=16 * 500)) for _ in range(40)]
    tr = tracegen.from_lists(reqs)
    B = 16
    caps = [1, 100, 5000, 30000]
    o = gu.oracle_run(tr, B, caps)
    assert o["n_distinct"] == o["n_access"] == 20000
    for with_outputs in (True, False):
        g = _run(tr, B, caps, with_outputs=with_outputs)
        for k in ("n_access", "n_distinct", "hits", "saved", "total_cost"):
            assert g[k] == o[k], (k, with_outputs)
        if with_outputs:
            gu.assert_same(g, o)
