"""The parity checks run against the checked build of the library.

Run by tests/test_gpu_checked.py in a process of its own (a process loads one
build): the checked build checks every index that comes from data another
stage or the caller wrote before using it, and reports a miss as
PTC_ERR_BOUNDS instead of touching memory.  Every call here must succeed and
match the oracle (the partitioned dedup of the id stage included, with and
without a prior-request hint)."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import paper_2609_28870_gb300 as ptc  # noqa: E402

ptc.use_checked_build()
assert b"checked" in ptc.lib().ptc_version(), ptc.lib().ptc_version()

import oracle  # noqa: E402
import tracegen  # noqa: E402
from tests.gpu_util import assert_same, oracle_run, to_gpu  # noqa: E402


NONE = 0xFFFFFFFF


def u32(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).cuda()


def pipeline(tr, B, caps, sessions):
    import torch
    tok, off, ts = to_gpu(tr)
    tok = tok[: tr.tokens.size] if tr.tokens.size else tok[:0]
    N = int(oracle.block_offsets(tr.req_tok_off, B)[-1])
    outs = {k: torch.empty(max(N, 1), dtype=torch.int32, device="cuda") for k in ("ids", "prev", "next", "dist")}
    outs["keys"] = torch.empty(2 * max(tr.tokens.size // B, 1), dtype=torch.int64, device="cuda")
    outs["req_blk_off"] = torch.empty(tr.n_req + 1, dtype=torch.int64, device="cuda")
    kw = dict(req_session=u32(tr.req_session), n_session=int(tr.req_session.max()) + 1) if sessions else {}
    res = ptc.ptc_pipeline(tok, off, ts, B, caps, outputs=outs, **kw)
    g = dict(res, req_blk_off=ptc.u64(outs["req_blk_off"]))
    for k in ("ids", "prev", "next", "dist"):
        g[k] = ptc.u32(outs[k])[:N]
    return g, outs


def main():
    cases = [(tracegen.tiny(s, n_sessions=1 + s % 9, vocab=2 + s % 3, max_seg=5 + 3 * s), 1 + s % 4) for s in range(8)]
    cases += [(tracegen.make(0), 16), (tracegen.make(1, max_requests=3000), 16), (tracegen.make(2, max_requests=60), 64)]
    for tr, B in cases:
        ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
        if ids.size == 0:
            continue
        caps = tracegen.capacity_grid(1, D + 2, 12)
        o = oracle_run(tr, B, caps)
        for sessions in (False, True):
            g, outs = pipeline(tr, B, caps, sessions)
            assert_same(g, o)
        off = outs["req_blk_off"]
        N = ids.size
        keys = outs["keys"].view(-1, 2)[:N]
        prior = u32(np.asarray([NONE] + list(range(tr.n_req - 1)), np.uint32)[: tr.n_req])
        for hint in ((None, None), (off, prior)):
            pid, pd = ptc.ptc_assign_ids_ex(keys, ptc.PTC_IDS_PARTITIONED, *hint)
            assert pd == D and np.array_equal(ptc.u32(pid), ids)
        bel = ptc.ptc_belady_curves(outs["prev"][:N], off, B, caps)
        h, s, raw = oracle.belady_curves(ids, oracle.block_offsets(tr.req_tok_off, B), B, caps)
        assert bel["hits"] == h and bel["saved"] == s and bel["raw_hits"] == raw
        ses = tr.req_session.astype(np.uint32)
        S = int(ses.max()) + 1
        sl = ptc.ptc_session_lru_curves(outs["ids"][:N], D, off, u32(ses), S, B, caps)
        h2, s2 = oracle.session_lru_curves(ids, oracle.block_offsets(tr.req_tok_off, B), ses, S, B, caps)
        assert sl["hits"] == h2 and sl["saved"] == s2
        for order, res in ((1, 0), (0, 1), (1, 1)):
            vd = ptc.ptc_stack_distance_variant(outs["prev"][:N], off, order, res)
            want = oracle.sd_variant(ids, D, oracle.block_offsets(tr.req_tok_off, B), order, res)
            assert np.array_equal(ptc.u32(vd), want)
    print("checked build: all calls clean and equal to the oracle")


if __name__ == "__main__":
    main()
