"""Trace statistics (Sec. 4.1-4.3, App. B) on the GPU against the oracle,
through the C ABI: every histogram, count and reach value bit-exact.  The GPU
side computes its ids, prev, next and stack distances itself (the pipeline);
the oracle derives its statistics from its own exact ids and distances."""
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


def _sess(sess, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(sess, dtype=np.uint32).view(np.int32)).to(device)


def gpu_stats(tr, B, caps=None, ts=None, sess=None, n_session=None, with_dist=True):
    """The GPU pipeline on the trace, then ptc_trace_stats on its arrays."""
    import torch
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util
    tok, off, ts_d = gpu_util.to_gpu(tr)
    tok = tok[: tr.tokens.size] if tr.tokens.size else tok[:0]
    out = ptc.pipeline(tok, off, ts_d, B, [1])
    ts_arr = tr.req_ts_us if ts is None else np.asarray(ts, dtype=np.int64)
    ses = tr.req_session if sess is None else np.asarray(sess)
    ns = tr.n_sessions if n_session is None else n_session
    ts_t = torch.from_numpy(np.ascontiguousarray(ts_arr, dtype=np.int64)).cuda()
    st = ptc.ptc_trace_stats(out["ids"], out["prev"], out["next"], out["n_distinct"], out["req_blk_off"], ts_t,
                             _sess(ses), ns, dist=out["dist"] if with_dist else None, caps=caps)
    return st


def oracle_stats(tr, B, caps=None, ts=None, sess=None, n_session=None, with_dist=True):
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    off = oracle.block_offsets(tr.req_tok_off, B)
    sd = oracle.sd_fenwick(oracle.reuse(ids, D)[0]) if with_dist else None
    return oracle.trace_stats(ids, D, off, tr.req_ts_us if ts is None else ts,
                              tr.req_session if sess is None else sess,
                              tr.n_sessions if n_session is None else n_session, sd, caps)


def assert_same_stats(g, o, with_reach=True):
    for k in oracle.STAT_SHAPES:
        assert g[k].shape == o[k].shape and np.array_equal(g[k], o[k]), k
    for k in oracle.STAT_SCALARS:
        assert g[k] == o[k], k
    if with_reach:
        assert np.array_equal(g["reach"], o["reach"])


def test_worked_example():
    gj = json.load(open(os.path.join(GOLDEN, "trace_stats_example.json")))
    tr = tracegen.from_lists(gj["requests"], ts=gj["ts_us"], sessions=gj["sessions"])
    B, caps = gj["block_size"], gj["capacities"]
    g = gpu_stats(tr, B, caps, n_session=gj["n_session"])
    assert_same_stats(g, oracle_stats(tr, B, caps, n_session=gj["n_session"]))
    assert g["reach"].tolist() == gj["expect"]["reach"] and g["blocks"].tolist() == gj["expect"]["blocks"]


@pytest.mark.parametrize("seed", range(24))
def test_tiny_random_traces(seed):
    rng = np.random.default_rng(9000 + seed)
    B = int(rng.choice([1, 2, 3, 4, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 12)), max_turns=int(rng.integers(1, 9)),
                       vocab=int(rng.integers(2, 6)))
    ts = np.cumsum(rng.choice([0, 1, 7, 1000, 3_000_000, 2**40], size=tr.n_req)).astype(np.int64)
    ns = int(tr.req_session.max()) + 1 + int(rng.integers(0, 3))  # some labels unused
    caps = np.unique(rng.integers(1, 40, size=int(rng.integers(1, 12)))).astype(np.uint64)
    g = gpu_stats(tr, B, caps, ts=ts, n_session=ns)
    assert_same_stats(g, oracle_stats(tr, B, caps, ts=ts, n_session=ns))


def test_without_distances():
    tr = tracegen.tiny(3, n_sessions=7)
    g = gpu_stats(tr, 2, with_dist=False)
    o = oracle_stats(tr, 2, with_dist=False)
    assert_same_stats(g, o, with_reach=False)
    assert int(g["dist_log2"].sum()) == 0 and "reach" not in g


def test_tiny_conversational_workload_full():
    tr = tracegen.make(0)
    caps = tracegen.workload_grid(0, 135_640)
    g = gpu_stats(tr, 16, caps)
    assert_same_stats(g, oracle_stats(tr, 16, caps))


def test_chat_workload_full_size():
    """The chat workload (~154M tokens, ~9.6M accesses) on its 64-point grid."""
    tr = tracegen.make(1)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(1, D)
    g = gpu_stats(tr, 16, caps)
    off = oracle.block_offsets(tr.req_tok_off, 16)
    sd = oracle.sd_fenwick(oracle.reuse(ids, D)[0])
    o = oracle.trace_stats(ids, D, off, tr.req_ts_us, tr.req_session, tr.n_sessions, sd, caps)
    assert_same_stats(g, o)
    # every category is populated on this workload
    assert np.all(g["blocks"] > 0)


def test_long_requests_span_many_tiles():
    """Requests of thousands of blocks (several 2048-access tiles each) next
    to empty and one-block requests, one long session and many short ones."""
    rng = np.random.default_rng(11)
    base = rng.integers(0, 50, size=40_000).tolist()
    reqs, sess, ts = [], [], []
    for j in range(12):
        reqs.append(base[: 3000 * (j + 1) // 1])
        sess.append(0)
        ts.append(1000 * j)
        reqs.append([])
        sess.append(1 + j)
        ts.append(1000 * j + 1)
        reqs.append([int(rng.integers(0, 3))])
        sess.append(13 + j % 2)
        ts.append(1000 * j + 2)
    tr = tracegen.from_lists(reqs, ts=ts, sessions=sess)
    caps = [1, 2, 100, 3000, 40_000]
    g = gpu_stats(tr, 1, caps)
    assert_same_stats(g, oracle_stats(tr, 1, caps))


def test_empty_and_degenerate_traces():
    # no full block anywhere: N = 0; sessions still counted
    tr = tracegen.from_lists([[1], [], [2, 3]], ts=[0, 5, 9], sessions=[0, 1, 0])
    g = gpu_stats(tr, 4, n_session=3)
    assert_same_stats(g, oracle_stats(tr, 4, n_session=3), with_reach=False)
    assert g["n_access"] == 0 and g["n_sessions"] == 2 and g["n_multi_sessions"] == 1
    # one access
    tr = tracegen.from_lists([[7, 7]], ts=[3], sessions=[0])
    g = gpu_stats(tr, 2, [1])
    assert_same_stats(g, oracle_stats(tr, 2, [1]))
    assert g["blocks"].tolist() == [0, 0, 1] and g["reach"].tolist() == [0]
    # every request the same, one session per request (a template: single-turn)
    tr = tracegen.from_lists([[4, 5, 6, 7]] * 9, ts=list(range(9)), sessions=list(range(9)))
    g = gpu_stats(tr, 2, [1, 2])
    assert_same_stats(g, oracle_stats(tr, 2, [1, 2]))
    assert g["blocks"].tolist() == [0, 0, 2] and g["freq"][2, 9] == 2


def test_error_statuses():
    import torch
    import paper_2609_28870_gb300 as ptc
    from tests import gpu_util
    tr = tracegen.from_lists([[1, 2], [1, 3], [1, 2, 4]], ts=[0, 5, 9], sessions=[0, 1, 0])
    tok, off, ts = gpu_util.to_gpu(tr)
    out = ptc.pipeline(tok[: tr.tokens.size], off, ts, 1, [1])
    args = (out["ids"], out["prev"], out["next"], out["n_distinct"], out["req_blk_off"])
    bad_ts = torch.tensor([0, 9, 5], dtype=torch.int64, device="cuda")
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_trace_stats(*args, bad_ts, _sess([0, 1, 0]), 2)
    assert e.value.name == "PTC_ERR_UNSORTED"
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_trace_stats(*args, ts, _sess([0, 2, 0]), 2)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    # an id at or above n_distinct
    ids = out["ids"].clone()
    ids[1] = out["n_distinct"]
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_trace_stats(ids, *args[1:], ts, _sess([0, 1, 0]), 2)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    # a prev that points forward
    prev = out["prev"].clone()
    prev[0] = 3
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_trace_stats(args[0], prev, *args[2:], ts, _sess([0, 1, 0]), 2)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    # still usable afterwards
    g = ptc.ptc_trace_stats(*args, ts, _sess([0, 1, 0]), 2)
    assert g["n_access"] == 7 and g["n_reuse"] == 7 - out["n_distinct"]
    assert_same_stats(g, oracle_stats(tr, 1, n_session=2, with_dist=False), with_reach=False)
