"""ptc_belady_curves (Belady's offline optimum, Sec. 3.2) against the
oracle's direct MIN simulation per capacity: prefix-counted hits, 128-bit
compute saved and raw hits, bit-exact, on hand-made and tiny random traces
at every capacity from 1 to D + 1, the tiny conversational workload and the
chat workload on their grids, and reuse arrays with short repeats that make
the run pieces meet themselves."""
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


def _u32(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).cuda()


def _check_ids(ids, off, B, caps, kinds=((1, oracle.F_LIN, oracle.F_ATTN),)):
    import paper_2609_28870_gb300 as ptc
    ids = np.asarray(ids, dtype=np.uint32)
    D = int(ids.max()) + 1 if ids.size else 0
    prev, _ = oracle.reuse(ids, D)
    for kind, f_lin, f_attn in kinds:
        h, s, raw = oracle.belady_curves(ids, off, B, caps, kind, f_lin, f_attn)
        g = ptc.ptc_belady_curves(_u32(prev), ptc.to_device_u64(np.asarray(off, np.uint64)), B, caps, kind, f_lin,
                                  f_attn)
        assert g["raw_hits"] == raw, kind
        assert g["hits"] == h, kind
        assert g["saved"] == s, kind


def test_worked_example_and_hand_traces():
    # the survey's worked example (B = 2) and traces built to hit each branch
    reqs = [[1, 2, 3, 4, 5], [1, 2, 7, 8], [1, 2, 3, 4, 5, 6, 9, 9], [3, 4, 1, 2], [1, 2, 7, 8, 0, 0]]
    tr = tracegen.from_lists(reqs)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 2)
    _check_ids(ids, oracle.block_offsets(tr.req_tok_off, 2), 2, np.arange(1, D + 2, dtype=np.uint64),
               ((0, 0, 0), (1, 1, 1), (2, 0, 1)))


@pytest.mark.parametrize("seed", range(24))
def test_tiny_random_traces(seed):
    rng = np.random.default_rng(1200 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 14)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 60)))
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    if ids.size == 0:
        return
    _check_ids(ids, oracle.block_offsets(tr.req_tok_off, B), B, np.arange(1, D + 2, dtype=np.uint64),
               ((0, 0, 0), (1, 3, 5), (2, 0, 7)))


@pytest.mark.parametrize("seed", range(8))
def test_short_repeats_and_long_runs(seed):
    """Id sequences outside prefix traces: periodic re-reads (runs that meet
    their own previous accesses), immediate repeats, and runs longer than the
    1,024 steps simulated together."""
    rng = np.random.default_rng(77 + seed)
    parts = []
    for _ in range(6):
        kind = rng.integers(0, 4)
        if kind == 0:
            per = int(rng.integers(1, 5))
            parts.append(np.tile(rng.integers(0, 50, per), int(rng.integers(2, 40))))
        elif kind == 1:
            parts.append(np.repeat(rng.integers(0, 50, 3), int(rng.integers(1, 5))))
        elif kind == 2:
            base = np.arange(int(rng.integers(1000, 3000)))
            parts.append(np.concatenate([base, rng.integers(0, 50, 7), base]))
        else:
            parts.append(rng.integers(0, 60, int(rng.integers(10, 300))))
    ids = np.concatenate(parts).astype(np.uint32)
    _, ids = np.unique(ids, return_inverse=True)  # dense ids
    cuts = np.sort(rng.choice(np.arange(1, ids.size), size=5, replace=False))
    off = np.concatenate([[0], cuts, [ids.size]]).astype(np.uint64)
    D = int(ids.max()) + 1
    caps = np.unique(np.concatenate([np.arange(1, 12), tracegen.capacity_grid(12, D + 1, 20)])).astype(np.uint64)
    _check_ids(ids.astype(np.uint32), off, 1, caps, ((0, 0, 0), (1, 2, 3)))


def test_tiny_conversational_workload():
    tr = tracegen.make(0)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    _check_ids(ids, oracle.block_offsets(tr.req_tok_off, 16), 16, tracegen.workload_grid(0, D))


def test_chat_workload_full():
    tr = tracegen.make(1)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(1, D)
    pick = np.arange(0, len(caps), 4)  # 16 of the 64 grid points for the oracle's time
    import paper_2609_28870_gb300 as ptc
    off = oracle.block_offsets(tr.req_tok_off, 16)
    prev, _ = oracle.reuse(ids, D)
    h, s, raw = oracle.belady_curves(ids, off, 16, caps[pick])
    g = ptc.ptc_belady_curves(_u32(prev), ptc.to_device_u64(off), 16, caps)
    assert [g["hits"][p] for p in pick] == h and [g["saved"][p] for p in pick] == s
    assert [g["raw_hits"][p] for p in pick] == raw
    # all 64 points: monotone, at least LRU's hits, N - D at D
    lru = oracle.curves_from_dist(oracle.sd_fenwick(prev), off, 16, caps)[0]
    assert all(a <= b for a, b in zip(g["hits"], g["hits"][1:]))
    assert all(b >= l for b, l in zip(g["raw_hits"], lru))
    assert g["hits"][-1] == ids.size - D


def test_errors():
    import paper_2609_28870_gb300 as ptc
    off = ptc.to_device_u64(np.array([0, 3], np.uint64))
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_belady_curves(_u32([oracle.NONE, 1, 0]), off, 1, [1, 2])  # prev[1] = 1 is not earlier
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_belady_curves(_u32([oracle.NONE, 0, 1]), off, 1, [2, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
    bad_off = ptc.to_device_u64(np.array([0, 2], np.uint64))
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_belady_curves(_u32([oracle.NONE, 0, 1]), bad_off, 1, [1, 2])
    assert e.value.name == "PTC_ERR_INVALID_ARG"
