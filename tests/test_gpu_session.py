"""ptc_session_lru_curves (session-level LRU eviction, Sec. 5.3) against the
oracle's direct per-capacity simulation, bit-exact: hits and 128-bit compute
saved on the hand-worked example, tiny random traces at every capacity from 1
to D + 2, the tiny conversational workload and a prefix of the chat workload
on their grids, and id sequences that repeat blocks inside a request."""
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


def _u32(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).cuda()


def _check(ids, off, ses, S, B, caps, kinds=((1, oracle.F_LIN, oracle.F_ATTN),)):
    import paper_2609_28870_gb300 as ptc
    ids = np.asarray(ids, dtype=np.uint32)
    D = int(ids.max()) + 1
    for kind, f_lin, f_attn in kinds:
        h, s = oracle.session_lru_curves(ids, off, ses, S, B, caps, kind, f_lin, f_attn)
        g = ptc.ptc_session_lru_curves(_u32(ids), D, ptc.to_device_u64(np.asarray(off, np.uint64)), _u32(ses), S, B,
                                       caps, kind, f_lin, f_attn)
        assert g["hits"] == h, kind
        assert g["saved"] == s, kind


def test_hand_worked_example():
    with open(os.path.join(GOLDEN, "session_lru_example.json")) as f:
        g = json.load(f)
    tr = tracegen.from_lists(g["requests"], sessions=g["sessions"])
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 1)
    import paper_2609_28870_gb300 as ptc
    out = ptc.ptc_session_lru_curves(_u32(ids), D, ptc.to_device_u64(oracle.block_offsets(tr.req_tok_off, 1)),
                                     _u32(g["sessions"]), 2, 1, np.asarray(g["capacities"], np.uint64),
                                     oracle.COST_UNIFORM)
    assert out["hits"] == g["hits"] and out["saved"] == g["hits"]


@pytest.mark.parametrize("seed", range(24))
def test_tiny_random_traces(seed):
    rng = np.random.default_rng(5000 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 12)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 60)))
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    if ids.size == 0:
        return
    ses = tr.req_session.astype(np.uint32)
    _check(ids, oracle.block_offsets(tr.req_tok_off, B), ses, int(ses.max()) + 1, B,
           np.arange(1, D + 3, dtype=np.uint64), ((0, 0, 0), (1, 3, 5), (2, 0, 7)))


@pytest.mark.parametrize("seed", range(6))
def test_repeated_blocks_inside_requests(seed):
    """Id sequences outside prefix traces: a request may touch a block twice."""
    rng = np.random.default_rng(600 + seed)
    n = 400
    ids = rng.integers(0, 40, n).astype(np.uint32)
    _, ids = np.unique(ids, return_inverse=True)
    cuts = np.sort(rng.choice(np.arange(1, n), size=30, replace=False))
    off = np.concatenate([[0], cuts, [n]]).astype(np.uint64)
    ses = rng.integers(0, 5, off.size - 1).astype(np.uint32)
    D = int(ids.max()) + 1
    _check(ids.astype(np.uint32), off, ses, 5, 1, np.arange(1, D + 3, dtype=np.uint64), ((0, 0, 0), (1, 2, 3)))


def test_tiny_conversational_workload():
    tr = tracegen.make(0)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    _check(ids, oracle.block_offsets(tr.req_tok_off, 16), tr.req_session.astype(np.uint32), tr.n_sessions, 16,
           tracegen.workload_grid(0, D))


def test_chat_workload_prefix():
    tr = tracegen.make(1, max_requests=4000)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    _check(ids, oracle.block_offsets(tr.req_tok_off, 16), tr.req_session.astype(np.uint32), tr.n_sessions, 16,
           tracegen.workload_grid(1, D))


def test_errors():
    import paper_2609_28870_gb300 as ptc
    off = ptc.to_device_u64(np.array([0, 2, 3], np.uint64))
    with pytest.raises(ptc.PtcError) as e:  # a label at n_session
        ptc.ptc_session_lru_curves(_u32([0, 1, 0]), 2, off, _u32([0, 2]), 2, 1, [1, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    with pytest.raises(ptc.PtcError) as e:  # an id at n_distinct
        ptc.ptc_session_lru_curves(_u32([0, 2, 0]), 2, off, _u32([0, 1]), 2, 1, [1, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    with pytest.raises(ptc.PtcError) as e:  # capacities not ascending
        ptc.ptc_session_lru_curves(_u32([0, 1, 0]), 2, off, _u32([0, 1]), 2, 1, [2, 1])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
