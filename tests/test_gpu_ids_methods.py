"""The id stage (ptc_assign_ids) against the oracle's exact ids, bit-exact.
The keys come from the oracle's own prefix hash, so this checks the id stage
alone: tiny traces, workload prefixes, all-distinct keys (the table's largest
fill), one key repeated, and a key that is not a field element."""
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


def _keys(keys_np):
    import paper_2609_28870_gb300 as ptc
    return ptc.to_device_u64(np.ascontiguousarray(keys_np).reshape(-1))


def _check_all(tr, B, seed=0):
    import paper_2609_28870_gb300 as ptc
    want, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    keys = _keys(oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, seed)).view(-1, 2)
    ids, d = ptc.ptc_assign_ids(keys)
    assert d == D
    assert np.array_equal(ptc.u32(ids), want)


@pytest.mark.parametrize("seed", range(12))
def test_tiny_traces(seed):
    rng = np.random.default_rng(7000 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 14)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 50)))
    _check_all(tr, B, seed)


@pytest.mark.parametrize("workload,requests,B", [(0, None, 16), (1, 3000, 16), (2, 150, 16), (2, 150, 64)])
def test_workloads(workload, requests, B):
    _check_all(tracegen.make(workload, max_requests=requests), B)


def test_all_distinct_and_all_equal_keys():
    """Every key distinct (the table's largest fill), and one key repeated."""
    import paper_2609_28870_gb300 as ptc
    rng = np.random.default_rng(5)
    distinct = rng.integers(0, (1 << 61) - 1, size=(20000, 2), dtype=np.uint64)
    same = np.repeat(distinct[:1], 5000, axis=0)
    for k, want_d in ((distinct, 20000), (same, 1)):
        ids, d = ptc.ptc_assign_ids(_keys(k).view(-1, 2))
        assert d == want_d
        got = ptc.u32(ids)
        if want_d == 1:
            assert not got.any()
        else:
            assert np.array_equal(got, np.arange(20000, dtype=np.uint32))


def test_invalid_key():
    import paper_2609_28870_gb300 as ptc
    bad = _keys(np.array([[1, 2], [(1 << 61) - 1, 4]], dtype=np.uint64)).view(-1, 2)  # not a field element
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_assign_ids(bad)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
