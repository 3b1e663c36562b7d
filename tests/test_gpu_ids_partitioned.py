"""The partitioned dedup of the id stage (ptc_assign_ids_ex with
PTC_IDS_PARTITIONED) against the oracle's exact ids, bit-exact, next to the
hash-table method on the same keys.

The partitioned method moves the keys to settle into 65,536 partitions by 16
bits of h0 and deduplicates each partition in shared memory; a partition with
more distinct keys than its shared table holds makes the call redo the stage
with the full hash table.  Covered: tiny traces and workload prefixes (keys
from the oracle's prefix hash, ids from its exact trie), with and without the
prior-request hint; random keys over several level-1 CTAs and several
level-2 tiles per bucket; ragged sizes around the warp and round widths; a
few keys repeated tens of thousands of times (partitions larger than one
pass of the dedup CTA); every key in one partition (the fallback); and a key
that is not a field element."""
import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu
NONE = 0xFFFFFFFF
P61 = (1 << 61) - 1


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_28870_gb300 as ptc
    ptc.lib()


def _keys(keys_np):
    import paper_2609_28870_gb300 as ptc
    return ptc.to_device_u64(np.ascontiguousarray(keys_np, dtype=np.uint64).reshape(-1)).view(-1, 2)


def _dev_u32(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).cuda()


def first_occurrence_ids(k):
    """Ids by definition: equal keys share an id, numbered in order of first
    occurrence."""
    v = np.ascontiguousarray(k, dtype=np.uint64).view(np.dtype((np.void, 16))).ravel()
    _, first, inv = np.unique(v, return_index=True, return_inverse=True)
    rank = np.empty(len(first), dtype=np.int64)
    rank[np.argsort(first, kind="stable")] = np.arange(len(first))
    return rank[inv.ravel()].astype(np.uint32), len(first)


def prior_by_session(labels):
    last, out = {}, []
    for r, s in enumerate(labels):
        out.append(last.get(int(s), NONE))
        last[int(s)] = r
    return np.asarray(out, dtype=np.uint32)


def _check_methods(keys, want, D, blk=None, prior=None):
    import paper_2609_28870_gb300 as ptc
    for method in (ptc.PTC_IDS_PARTITIONED, ptc.PTC_IDS_TABLE):
        ids, d = ptc.ptc_assign_ids_ex(keys, method, blk, prior)
        assert d == D, method
        assert np.array_equal(ptc.u32(ids), want), method


def _check_trace(tr, B, seed=0):
    import paper_2609_28870_gb300 as ptc
    want, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    keys = _keys(oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, seed))
    _check_methods(keys, want, D)
    blk = ptc.to_device_u64(oracle.block_offsets(tr.req_tok_off, B))
    rng = np.random.default_rng(seed)
    rnd = np.full(tr.n_req, NONE, np.uint32)
    for r in range(1, tr.n_req):
        if rng.random() < 0.9:
            rnd[r] = rng.integers(0, r)
    for prior in (prior_by_session(tr.req_session), rnd):
        _check_methods(keys, want, D, blk, _dev_u32(prior))


@pytest.mark.parametrize("seed", range(10))
def test_tiny_traces(seed):
    rng = np.random.default_rng(9100 + seed)
    B = int(rng.choice([1, 2, 3, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 14)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 50)))
    _check_trace(tr, B, seed)


@pytest.mark.parametrize("workload,requests,B", [(0, None, 16), (1, 3000, 16), (2, 150, 16), (2, 150, 64),
                                                 (3, 400, 16)])
def test_workload_prefixes(workload, requests, B):
    _check_trace(tracegen.make(workload, max_requests=requests), B)


def _random_keys(rng, n_distinct, n, zipf=None):
    pool = rng.integers(0, P61, size=(n_distinct, 2), dtype=np.uint64)
    if zipf is None:
        pick = rng.integers(0, n_distinct, size=n)
    else:
        pick = np.minimum(rng.zipf(zipf, size=n) - 1, n_distinct - 1)
    return pool[pick]


def test_random_keys_many_ctas_and_tiles():
    """3M keys over 2M distinct: every level-1 CTA range and several level-2
    tiles per bucket (about 11,700 records each) are used."""
    rng = np.random.default_rng(31)
    k = _random_keys(rng, 2_000_000, 3_000_000)
    want, D = first_occurrence_ids(k)
    _check_methods(_keys(k), want, D)


@pytest.mark.parametrize("n", [1, 2, 31, 32, 33, 255, 1023, 1024, 1025, 4097, 70001])
def test_ragged_sizes(n):
    rng = np.random.default_rng(n)
    k = _random_keys(rng, max(1, n // 2), n)
    want, D = first_occurrence_ids(k)
    _check_methods(_keys(k), want, D)


def test_hot_keys():
    """Five keys repeated 40,000 times each among 100,000 distinct ones, in a
    random order: their partitions take many passes of the dedup CTA."""
    rng = np.random.default_rng(77)
    hot = rng.integers(0, P61, size=(5, 2), dtype=np.uint64)
    cold = rng.integers(0, P61, size=(100_000, 2), dtype=np.uint64)
    k = np.concatenate([np.repeat(hot, 40_000, axis=0), cold])
    k = k[rng.permutation(len(k))]
    want, D = first_occurrence_ids(k)
    _check_methods(_keys(k), want, D)


def test_zipf_repeats():
    rng = np.random.default_rng(78)
    k = _random_keys(rng, 400_000, 1_500_000, zipf=1.3)
    want, D = first_occurrence_ids(k)
    _check_methods(_keys(k), want, D)


def test_one_partition_overflows_to_the_full_table():
    """10,000 distinct keys that all share h0 bits 45..60 fall in one
    partition, more than its shared table holds: the call redoes the stage
    with the full table and still gives exact ids."""
    rng = np.random.default_rng(79)
    low = rng.integers(0, 1 << 45, size=10_000, dtype=np.uint64)
    h0 = (np.uint64(0x1234) << np.uint64(45)) | low
    h1 = rng.integers(0, P61, size=10_000, dtype=np.uint64)
    distinct = np.stack([h0, h1], axis=1)
    k = distinct[rng.integers(0, 10_000, size=30_000)]
    want, D = first_occurrence_ids(k)
    assert D > 6144
    _check_methods(_keys(k), want, D)


def test_invalid_key():
    import paper_2609_28870_gb300 as ptc
    bad = _keys(np.array([[1, 2], [P61, 4]], dtype=np.uint64))  # not a field element
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_assign_ids_ex(bad, ptc.PTC_IDS_PARTITIONED)
    assert e.value.name == "PTC_ERR_INVALID_ARG"


def test_unknown_method():
    import paper_2609_28870_gb300 as ptc
    k = _keys(np.array([[1, 2]], dtype=np.uint64))
    with pytest.raises(ptc.PtcError) as e:
        ptc.ptc_assign_ids_ex(k, 7)
    assert e.value.name == "PTC_ERR_INVALID_ARG"
