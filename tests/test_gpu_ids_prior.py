"""The prior-request hint of the id stage against the oracle's exact ids.

ptc_assign_ids_prior takes, for every request, an earlier request whose
blocks it is likely to repeat (a turn of a session re-sends that session's
previous context, Sec. 2.3) and skips the table for the blocks that repeat
it.  The ids must not depend on the hint: for every hint with prior[r] < r
(or none) they equal the oracle's exact first-occurrence ids.  The hints here
are the sessions' previous requests (the one the pipeline uses), a random
earlier request, the request just before, no hint at all, and a request that
shares only the root blocks.  ptc_session_prior is checked against its
definition, and ptc_pipeline with sessions against the whole oracle."""
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
    import paper_2609_28870_gb300 as ptc
    ptc.lib()


def prior_by_definition(labels):
    """The latest earlier request with the same session label."""
    last, out = {}, []
    for r, s in enumerate(labels):
        out.append(last.get(int(s), NONE))
        last[int(s)] = r
    return np.asarray(out, dtype=np.uint32)


def _dev_u32(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).cuda()


def hints(tr, B, rng):
    """Several prior arrays for one trace, every one valid (prior[r] < r)."""
    R = tr.n_req
    off = oracle.block_offsets(tr.req_tok_off, B)
    out = {"session": prior_by_definition(tr.req_session), "none": np.full(R, NONE, np.uint32),
           "previous": np.asarray([NONE] + list(range(R - 1)), np.uint32)[:R]}
    rnd = np.full(R, NONE, np.uint32)
    for r in range(1, R):
        if rng.random() < 0.9:
            rnd[r] = rng.integers(0, r)
    out["random"] = rnd
    # the earliest request whose first block equals this one's (shares the root only, in general)
    ids, _ = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    root = np.full(R, NONE, np.uint32)
    seen = {}
    for r in range(R):
        if off[r + 1] > off[r]:
            first = int(ids[off[r]])
            root[r] = seen.get(first, NONE)
            seen.setdefault(first, r)
    out["same_root"] = root
    return out


def _check(tr, B, seed=0, rng=None):
    import paper_2609_28870_gb300 as ptc
    rng = rng or np.random.default_rng(seed)
    want, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    keys = ptc.to_device_u64(oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, seed).reshape(-1)).view(-1, 2)
    blk = ptc.to_device_u64(oracle.block_offsets(tr.req_tok_off, B))
    for name, pr in hints(tr, B, rng).items():
        ids, d = ptc.ptc_assign_ids_prior(keys, blk, _dev_u32(pr))
        assert d == D, name
        assert np.array_equal(ptc.u32(ids), want), name


def test_session_prior_definition():
    import paper_2609_28870_gb300 as ptc
    rng = np.random.default_rng(1)
    for R, S in ((1, 1), (5, 2), (1000, 7), (50000, 70000), (200000, 300), (3, 1 << 31)):
        labels = rng.integers(0, S, size=R).astype(np.uint32)
        got = ptc.u32(ptc.ptc_session_prior(_dev_u32(labels), S))
        assert np.array_equal(got, prior_by_definition(labels)), (R, S)


def test_session_prior_label_out_of_range():
    import paper_2609_28870_gb300 as ptc
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_session_prior(_dev_u32([0, 3, 1]), 3)
    assert e.value.name == "PTC_ERR_INVALID_ARG"


@pytest.mark.parametrize("seed", range(16))
def test_tiny_traces_every_hint(seed):
    rng = np.random.default_rng(8000 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 14)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 50)))
    _check(tr, B, seed, rng)


@pytest.mark.parametrize("workload,requests,B", [(0, None, 16), (1, 3000, 16), (2, 150, 16), (2, 150, 64),
                                                 (3, 4000, 16)])
def test_workload_prefixes_every_hint(workload, requests, B):
    _check(tracegen.make(workload, max_requests=requests), B)


def test_hint_pointing_forward_is_rejected():
    import paper_2609_28870_gb300 as ptc
    tr = tracegen.from_lists([[1, 2, 3, 4], [1, 2, 3, 4, 5, 6]])
    keys = ptc.to_device_u64(oracle.prefix_hash(tr.tokens, tr.req_tok_off, 2, 0).reshape(-1)).view(-1, 2)
    blk = ptc.to_device_u64(oracle.block_offsets(tr.req_tok_off, 2))
    for bad in ([1, NONE], [0, 1], [NONE, 5]):
        with pytest.raises(ptc.PtcError) as e:
            ptc.ptc_assign_ids_prior(keys, blk, _dev_u32(bad))
        assert e.value.name == "PTC_ERR_INVALID_ARG", bad
    ids, d = ptc.ptc_assign_ids_prior(keys, blk, _dev_u32([NONE, 0]))
    assert d == 3 and ptc.u32(ids).tolist() == [0, 1, 0, 1, 2]


def test_hint_through_requests_without_blocks():
    """Chains that pass through requests with no full block, whose own hints
    are then read by the chain walk."""
    import paper_2609_28870_gb300 as ptc
    reqs = [[1, 2, 3, 4], [9], [1, 2, 3, 4, 5, 6], [], [1, 2, 3, 4, 5, 6, 7, 8]]
    tr = tracegen.from_lists(reqs)
    want, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 2)
    keys = ptc.to_device_u64(oracle.prefix_hash(tr.tokens, tr.req_tok_off, 2, 0).reshape(-1)).view(-1, 2)
    blk = ptc.to_device_u64(oracle.block_offsets(tr.req_tok_off, 2))
    for pr in ([NONE, 0, 1, 2, 3], [NONE, NONE, 0, NONE, 2], [NONE, 0, 0, 1, 3]):
        ids, d = ptc.ptc_assign_ids_prior(keys, blk, _dev_u32(pr))
        assert d == D and np.array_equal(ptc.u32(ids), want), pr


@pytest.mark.parametrize("seed", range(8))
def test_pipeline_with_sessions_tiny(seed):
    """ptc_pipeline with session labels: every output equals the oracle's."""
    import paper_2609_28870_gb300 as ptc
    from tests.gpu_util import assert_same, oracle_run, to_gpu
    rng = np.random.default_rng(9000 + seed)
    B = int(rng.choice([1, 2, 4, 16]))
    tr = tracegen.tiny(100 + seed, n_sessions=int(rng.integers(1, 12)), vocab=int(rng.integers(2, 5)),
                       max_seg=int(rng.integers(3, 40)))
    o = oracle_run(tr, B, np.arange(1, 40, dtype=np.uint64))
    tok, off, ts = to_gpu(tr)
    tok = tok[: tr.tokens.size] if tr.tokens.size else tok[:0]
    n_ses = int(tr.req_session.max()) + 1 if tr.n_req else 1
    outs = {k: ptc.torch.empty(max(o["n_access"], 1), dtype=ptc.torch.int32, device="cuda")
            for k in ("ids", "prev", "next", "dist")}
    outs["req_blk_off"] = ptc.torch.empty(tr.n_req + 1, dtype=ptc.torch.int64, device="cuda")
    res = ptc.ptc_pipeline(tok, off, ts, B, np.arange(1, 40, dtype=np.uint64), outputs=outs,
                           req_session=_dev_u32(tr.req_session), n_session=n_ses)
    n = res["n_access"]
    g = dict(res, req_blk_off=ptc.u64(outs["req_blk_off"]))
    for k in ("ids", "prev", "next", "dist"):
        g[k] = ptc.u32(outs[k])[:n]
    assert_same(g, o)


@pytest.mark.parametrize("workload,requests", [(0, None), (1, 4000), (3, 3000)])
def test_pipeline_with_sessions_workloads(workload, requests):
    import paper_2609_28870_gb300 as ptc
    from tests.gpu_util import assert_same, oracle_run, to_gpu
    tr = tracegen.make(workload, max_requests=requests)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(min(workload, 3), D)
    o = oracle_run(tr, 16, caps)
    tok, off, ts = to_gpu(tr)
    N = o["n_access"]
    outs = {k: ptc.torch.empty(N, dtype=ptc.torch.int32, device="cuda") for k in ("ids", "prev", "next", "dist")}
    outs["req_blk_off"] = ptc.torch.empty(tr.n_req + 1, dtype=ptc.torch.int64, device="cuda")
    res = ptc.ptc_pipeline(tok, off, ts, 16, caps, outputs=outs, req_session=_dev_u32(tr.req_session),
                           n_session=tr.n_sessions)
    g = dict(res, req_blk_off=ptc.u64(outs["req_blk_off"]))
    for k in ("ids", "prev", "next", "dist"):
        g[k] = ptc.u32(outs[k])
    assert_same(g, o)


def test_pipeline_session_label_out_of_range():
    import paper_2609_28870_gb300 as ptc
    from tests.gpu_util import to_gpu
    tr = tracegen.tiny(3, n_sessions=4)
    tok, off, ts = to_gpu(tr)
    bad = np.asarray(tr.req_session, np.uint32).copy()
    bad[-1] = 4
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_pipeline(tok[: tr.tokens.size], off, ts, 2, [1, 2], req_session=_dev_u32(bad), n_session=4)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
