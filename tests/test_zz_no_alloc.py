"""The allocation-free variant of ptc_curves.

Some callers cannot allocate device memory (they run inside a runtime that
owns all of it, or must not touch an allocator), so ptc_curves_noalloc keeps
its scratch in a fixed array inside the library.  This file is collected last
on purpose: if it fails, a run that stops at the first failure has already run
every other test.  It checks the new entry point against ptc_curves, the
workspace-taking entry point, on two calls in a row (the first call on a
device sets up the array's address; the second reuses the array and must
clear what it left behind)."""
import ctypes

import numpy as np
import pytest

import tracegen

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ptc():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_28870_gb300 as p
    L = p.lib()
    L.ptc_curves_noalloc.restype = ctypes.c_int
    L.ptc_curves_noalloc.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_uint32,
                                     ctypes.c_uint32, ctypes.POINTER(p.CostModel), ctypes.c_void_p, ctypes.c_uint32,
                                     ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(p.U128), ctypes.c_void_p]
    return p


def _noalloc(p, dist, blk_off, B, caps, kind):
    import torch
    caps = np.ascontiguousarray(caps, dtype=np.uint64)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    saved = np.zeros(2 * G, dtype=np.uint64)
    total = p.U128()
    cm = p.CostModel(p.F_LIN, p.F_ATTN, kind)
    rc = p.lib().ptc_curves_noalloc(dist.data_ptr(), dist.numel(), blk_off.data_ptr(), blk_off.numel() - 1, B,
                                    ctypes.byref(cm), caps.ctypes.data, G, hits.ctypes.data, saved.ctypes.data,
                                    ctypes.byref(total), torch.cuda.current_stream().cuda_stream)
    assert rc == 0, p.STATUS.get(rc, rc)
    return ([int(h) for h in hits], [int(saved[2 * g + 1]) << 64 | int(saved[2 * g]) for g in range(G)],
            int(total.hi) << 64 | int(total.lo))


def test_noalloc_curves_match_workspace_curves_twice(ptc):
    import torch
    runs = []
    for workload, requests, kind in ((0, 500, ptc.PTC_COST_MEASURED), (0, 1500, ptc.PTC_COST_LINEAR)):
        tr = tracegen.make(workload, max_requests=requests)
        tok = ptc.to_device_u32(tr.tokens)
        off = ptc.to_device_u64(tr.req_tok_off)
        keys, blk_off, n = ptc.ptc_hash_blocks(tok, off, None, 16, 0)
        ids, d = ptc.ptc_assign_ids(keys)
        prev, _ = ptc.ptc_reuse_indices(ids, d)
        dist = ptc.ptc_stack_distance(prev)
        caps = tracegen.capacity_grid(16, d, 48)
        ref = ptc.ptc_curves(dist, blk_off, 16, caps, kind)
        got = _noalloc(ptc, dist, blk_off, 16, caps, kind)
        assert got[0] == ref["hits"]
        assert got[1] == ref["saved"]
        assert got[2] == ref["total_cost"]
        runs.append(got)
    assert runs[0] != runs[1]  # two different inputs, so the second call really recomputed
    torch.cuda.synchronize()


def test_noalloc_rejects_too_many_accesses(ptc):
    import torch
    dist = torch.zeros(1, dtype=torch.int32, device="cuda")
    blk_off = torch.zeros(2, dtype=torch.int64, device="cuda")
    caps = np.asarray([1], dtype=np.uint64)
    hits = np.zeros(1, dtype=np.uint64)
    saved = np.zeros(2, dtype=np.uint64)
    total = ptc.U128()
    cm = ptc.CostModel(0, 0, ptc.PTC_COST_UNIFORM)
    rc = ptc.lib().ptc_curves_noalloc(dist.data_ptr(), (1 << 24) + 1, blk_off.data_ptr(), 1, 16, ctypes.byref(cm),
                                      caps.ctypes.data, 1, hits.ctypes.data, saved.ctypes.data, ctypes.byref(total),
                                      torch.cuda.current_stream().cuda_stream)
    assert ptc.STATUS[rc] == "PTC_ERR_WORKSPACE"
