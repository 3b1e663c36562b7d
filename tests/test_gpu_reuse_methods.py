"""Both sorts of the reuse stage (every (id, i), and the pieces of the
id-runs) against the oracle's prev / next, bit-exact."""
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


def _check_all(ids, D):
    import paper_2609_28870_gb300 as ptc
    want_p, want_n = oracle.reuse(ids, D)
    t = ptc.to_device_u32(ids)
    for m in (None, ptc.PTC_REUSE_AUTO, ptc.PTC_REUSE_SORT, ptc.PTC_REUSE_RUNS):
        p, n = ptc.ptc_reuse_indices(t, D, method=m)
        assert np.array_equal(ptc.u32(p), want_p), m
        assert np.array_equal(ptc.u32(n), want_n), m


@pytest.mark.parametrize("seed", range(16))
def test_tiny_traces(seed):
    rng = np.random.default_rng(3000 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 14)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 50)))
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    if ids.size:
        _check_all(ids, D)


@pytest.mark.parametrize("workload,requests", [(0, None), (1, 2500), (2, 120)])
def test_workloads(workload, requests):
    tr = tracegen.make(workload, max_requests=requests)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    _check_all(ids, D)


def test_hand_made_id_sequences():
    """Arbitrary dense ids (not in first-use order), overlapping and nested
    id-runs, a run re-read in pieces, one access, all equal, all distinct."""
    cases = [
        [0],
        [0, 0, 0, 0],
        list(range(50)),
        list(range(10)) + list(range(3, 7)) + list(range(10)) + [9, 8, 7],
        [5, 6, 7, 0, 1, 2, 3, 4, 5, 6, 7, 2, 3, 4],
        list(range(20, 40)) + list(range(0, 25)) + list(range(30, 45)) + list(range(10, 35)),
    ]
    for c in cases:
        ids = np.asarray(c, dtype=np.uint32)
        _check_all(ids, int(ids.max()) + 1)


def test_random_ids_fall_back_and_large_runs():
    rng = np.random.default_rng(5)
    ids = rng.integers(0, 5000, size=200000).astype(np.uint32)
    _check_all(ids, 5000)
    # long re-read runs over a large id space
    base = np.arange(300000, dtype=np.uint32)
    ids = np.concatenate([base, base[1000:250000], base[:5000], base[200000:300000]])
    _check_all(ids, 300000)


def test_ids_out_of_range_are_rejected():
    import paper_2609_28870_gb300 as ptc
    t = ptc.to_device_u32(np.asarray([0, 1, 2, 7, 3], dtype=np.uint32))
    for m in (ptc.PTC_REUSE_AUTO, ptc.PTC_REUSE_SORT, ptc.PTC_REUSE_RUNS):
        with pytest.raises(ptc.PtcError) as e:
            ptc.ptc_reuse_indices(t, 5, method=m)
        assert e.value.name == "PTC_ERR_INVALID_ARG"
