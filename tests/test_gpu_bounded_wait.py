"""Failure detection of the bounded device waits, with no GPU fault.

Kernels that wait on other CTAs (the decoupled look-back of stage a1's block
offsets) poll a bounded number of times and then give up with
PTC_ERR_TIMEOUT.  The test hook ptc_test_wait_polls makes those waits see no
predecessor as ready (a flag nothing sets) and give up after a few hundred
polls, so the give-up path runs for real: the call must return
PTC_ERR_TIMEOUT, nothing downstream may read through the unfinished offsets,
and the next call, with normal waits, must be bit-exact against the oracle on
the same device."""
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


def test_forced_give_up_then_exact_results():
    import torch

    import paper_2609_28870_gb300 as ptc
    from tests.gpu_util import to_gpu
    tr = tracegen.make(0, max_requests=1500)  # 1,500 requests: six 256-request tiles of the offsets scan
    B = 16
    tok, off, ts = to_gpu(tr)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
    caps = tracegen.workload_grid(0, D)
    L = ptc.lib()
    L.ptc_test_wait_polls(300)
    try:
        with pytest.raises(ptc.PtcError) as e:
            ptc.ptc_hash_blocks(tok, off, ts, B, 0)
        assert e.value.name == "PTC_ERR_TIMEOUT"
        with pytest.raises(ptc.PtcError) as e:
            ptc.ptc_pipeline(tok, off, ts, B, caps)
        assert e.value.name == "PTC_ERR_TIMEOUT"
    finally:
        L.ptc_test_wait_polls(0)
    torch.cuda.synchronize()  # the context is still usable
    keys, blk_off, n = ptc.ptc_hash_blocks(tok, off, ts, B, 0)
    assert n == ids.size
    assert np.array_equal(ptc.u64(blk_off), oracle.block_offsets(tr.req_tok_off, B))
    assert np.array_equal(ptc.u64(keys).reshape(-1, 2), oracle.prefix_hash(tr.tokens, tr.req_tok_off, B, 0))
    o = oracle.run(tr.tokens, tr.req_tok_off, B, caps)
    g = ptc.ptc_pipeline(tok, off, ts, B, caps)
    assert g["n_distinct"] == D and g["hits"] == o["hits"] and g["saved"] == o["saved"]
    assert g["total_cost"] == o["total_cost"]
