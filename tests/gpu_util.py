"""Helpers for the GPU parity tests: run the library on a trace and the
oracle on the same trace, returning numpy arrays."""
import numpy as np
import torch

import oracle
import paper_2609_28870_gb300 as ptc


def to_gpu(tr, device="cuda:0"):
    tok = ptc.to_device_u32(tr.tokens, device) if tr.tokens.size else torch.zeros(1, dtype=torch.int32, device=device)
    off = ptc.to_device_u64(tr.req_tok_off, device)
    ts = torch.from_numpy(np.ascontiguousarray(tr.req_ts_us)).to(device) if tr.n_req else None
    return tok, off, ts


def gpu_run(tr, B, caps, kind=oracle.COST_MEASURED, seed=0, f_lin=oracle.F_LIN, f_attn=oracle.F_ATTN):
    tok, off, ts = to_gpu(tr)
    tok = tok[: tr.tokens.size] if tr.tokens.size else tok[:0]
    out = ptc.pipeline(tok, off, ts, B, caps, kind=kind, seed=seed, f_lin=f_lin, f_attn=f_attn)
    res = dict(n_access=out["n_access"], n_distinct=out["n_distinct"], hits=out["hits"], saved=out["saved"],
               total_cost=out["total_cost"], caps=out["caps"])
    for k in ("ids", "prev", "next", "dist"):
        res[k] = ptc.u32(out[k])
    res["keys"] = ptc.u64(out["keys"]).reshape(-1, 2)
    res["req_blk_off"] = ptc.u64(out["req_blk_off"])
    return res


def oracle_run(tr, B, caps, kind=oracle.COST_MEASURED, f_lin=oracle.F_LIN, f_attn=oracle.F_ATTN, threads=None):
    return oracle.run(tr.tokens, tr.req_tok_off, B, caps, kind, f_lin, f_attn, threads)


def assert_same(g, o, caps_checked=True):
    assert g["n_access"] == o["n_access"]
    assert np.array_equal(g["req_blk_off"], o["req_blk_off"])
    assert g["n_distinct"] == o["n_distinct"]
    assert np.array_equal(g["ids"], o["ids"])
    assert np.array_equal(g["prev"], o["prev"])
    assert np.array_equal(g["next"], o["next"])
    assert np.array_equal(g["dist"], o["sd"])
    if caps_checked:
        assert g["hits"] == o["hits"]
        assert g["saved"] == o["saved"]
        assert g["total_cost"] == o["total_cost"]
