"""Both wavelet matrices of the stack-distance stage (over every access and
over runs) against the oracle's distances, bit-exact, on traces with short
and with long runs."""
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


def _ids_prev(tr, B):
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    prev, _ = oracle.reuse(ids, D)
    return ids, prev


def _all_methods(prev):
    import paper_2609_28870_gb300 as ptc
    p = ptc.to_device_u32(prev)
    return {m: ptc.u32(ptc.ptc_stack_distance(p, method=m)) for m in
            (ptc.PTC_SD_AUTO, ptc.PTC_SD_POINTS, ptc.PTC_SD_RUNS)}


@pytest.mark.parametrize("seed", range(20))
def test_methods_agree_on_tiny_traces(seed):
    rng = np.random.default_rng(7000 + seed)
    B = int(rng.choice([1, 2, 3, 4, 16]))
    tr = tracegen.tiny(seed, n_sessions=int(rng.integers(1, 14)), max_turns=7, vocab=int(rng.integers(2, 6)),
                       max_seg=int(rng.integers(3, 50)))
    ids, prev = _ids_prev(tr, B)
    if prev.size == 0:
        pytest.skip("no blocks")
    want = oracle.sd_mattson(ids)
    for m, got in _all_methods(prev).items():
        assert np.array_equal(got, want), m


@pytest.mark.parametrize("workload,requests", [(0, None), (1, 3000), (2, 150)])
def test_methods_agree_on_workloads(workload, requests):
    tr = tracegen.make(workload, max_requests=requests)
    _, prev = _ids_prev(tr, 16)
    want = oracle.sd_fenwick(prev)
    for m, got in _all_methods(prev).items():
        assert np.array_equal(got, want), m


def test_runs_edge_cases():
    """Hand-made reuse arrays: one access; all first accesses; one long
    context run; a window that is empty (prev = i - 1); alternating runs that
    break every access; a run cut by the window start."""
    N = oracle.NONE
    cases = [
        [N],
        [N] * 40,
        [N] * 10 + list(range(10)),
        [N, 0, 1, 2],
        [N, N, 1, 0, 3, 2, 5, 4],
        [N] * 6 + [2, 3, 4, 5] + [N, N] + [0, 1],
        [N] * 5 + [0, 1, 2] + [6, 7] + [3, 4],
    ]
    for prev in cases:
        prev = np.asarray(prev, dtype=np.uint32)
        # each case must be a reuse array: prev[i] < i, each value used once
        fin = prev[prev != N]
        assert len(set(fin.tolist())) == fin.size
        assert all(p < i for i, p in enumerate(prev.tolist()) if p != N)
        want = oracle.sd_fenwick(prev)
        for m, got in _all_methods(prev).items():
            assert np.array_equal(got, want), (prev.tolist(), m, got.tolist(), want.tolist())


def test_forced_runs_with_a_small_workspace_is_refused():
    import torch
    import paper_2609_28870_gb300 as ptc
    prev = np.full(5000, oracle.NONE, dtype=np.uint32)
    prev[1::2] = np.arange(0, 4999, 2, dtype=np.uint32)  # every access starts a run
    want = oracle.sd_fenwick(prev)
    p = ptc.to_device_u32(prev)
    L = ptc.lib()
    ws = torch.empty(L.ptc_stack_distance_workspace_bytes(prev.size), dtype=torch.uint8, device="cuda")
    # the automatic choice falls back to the matrix over accesses
    assert np.array_equal(ptc.u32(ptc.ptc_stack_distance(p, ws=ws)), want)
    dist = torch.empty(prev.size, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    rc = L.ptc_stack_distance_ex(p.data_ptr(), prev.size, dist.data_ptr(), ptc.PTC_SD_RUNS, ws.data_ptr(),
                                 ws.numel(), stream)
    assert ptc.STATUS[rc] == "PTC_ERR_WORKSPACE"
    big = torch.empty(L.ptc_stack_distance_ex_workspace_bytes(prev.size, ptc.PTC_SD_RUNS), dtype=torch.uint8,
                      device="cuda")
    rc = L.ptc_stack_distance_ex(p.data_ptr(), prev.size, dist.data_ptr(), ptc.PTC_SD_RUNS, big.data_ptr(),
                                 big.numel(), stream)
    assert rc == 0 and np.array_equal(ptc.u32(dist), want)
    rc = L.ptc_stack_distance_ex(p.data_ptr(), prev.size, dist.data_ptr(), 7, big.data_ptr(), big.numel(), stream)
    assert ptc.STATUS[rc] == "PTC_ERR_INVALID_ARG"


def test_many_runs_take_the_per_level_build():
    """More runs than one cluster's shared memory holds (131,072): the matrix
    over runs is built one level per launch; a random reuse array with short
    runs, forced onto the matrix over runs."""
    import torch
    import paper_2609_28870_gb300 as ptc
    rng = np.random.default_rng(11)
    ids = rng.integers(0, 60000, size=300000).astype(np.uint32)
    _, first = np.unique(ids, return_index=True)
    order = np.argsort(np.argsort(first))
    dense = np.empty_like(ids)
    remap = np.empty(ids.max() + 1, dtype=np.uint32)
    remap[np.unique(ids)] = order.astype(np.uint32)
    dense = remap[ids]
    prev, _ = oracle.reuse(dense, int(dense.max()) + 1)
    want = oracle.sd_fenwick(prev)
    p = ptc.to_device_u32(prev)
    got = ptc.u32(ptc.ptc_stack_distance(p, method=ptc.PTC_SD_RUNS))
    assert np.array_equal(got, want)
