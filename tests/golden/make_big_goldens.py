#!/usr/bin/env python3
"""Write tests/golden/big_configs.json: the oracle's results on the two
full-size traces that are too large for the oracle to run inside a GPU test.

    python tests/golden/make_big_goldens.py [--only agentic|mixed] [--threads N]

Entries (each one trace at one block size):
  agentic_B16, agentic_B32, agentic_B64, agentic_B256
      the agentic coding trace (seed 2, ~2.1B tokens) re-blocked at B = 16,
      32, 64 and 256 (the block-granularity study), on the token-denominated
      capacity grid: 16 x a 128-point grid from 0.1% to 100% of the distinct
      blocks at B = 16, as whole blocks of B;
  mixed_B16
      the mixed 24-hour trace (seed 3, ~10B tokens, ~624M block accesses) on
      its 128-point grid from 0.1% to 100% of the distinct blocks.

Each entry holds N, D, the SHA-256 of the trace's tokens and request offsets,
the SHA-256 of the oracle's ids, prev, next and stack distances (uint32,
little-endian), the capacity grid, hits and 128-bit compute saved at every
grid point from the oracle's distances by Mattson inclusion
(oracle.curves_from_dist), the total cost, and hits and compute saved by the
oracle's direct per-capacity LRU simulation (oracle.lru_curves) at a few grid
points.  Cost model: the measured shape (B f_lin + f_attn * positions
attended, f_lin = 6.6e9, f_attn = 786,432).

This script calls only oracle/ and tracegen/; no value here comes from the
GPU path.  The mixed trace needs about 55 GB of host memory while the oracle's
exact trie is built (40 GB of tokens plus the trie).
"""
from __future__ import annotations

import argparse
import gc
import hashlib
import json
import os
import resource
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import tracegen  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "big_configs.json")


def sha(a: np.ndarray) -> str:
    h = hashlib.sha256()
    mv = memoryview(np.ascontiguousarray(a)).cast("B")
    step = 1 << 28
    for i in range(0, len(mv), step):
        h.update(mv[i:i + step])
    return h.hexdigest()


def peak_gb() -> float:
    return resource.getrusage(resource.RUSAGE_SELF).ru_maxrss / 1e6


def token_grid(d16: int, B: int) -> np.ndarray:
    """Capacities in tokens (16 x a 0.1%-100% grid over the distinct blocks at
    B = 16), as whole blocks of B; equal points after rounding collapse."""
    base = tracegen.capacity_grid(max(1, round(0.001 * d16)), d16, 128).astype(np.uint64)
    return np.unique(np.maximum(np.uint64(1), (np.uint64(16) * base) // np.uint64(B)))


def entry(ids, D, req_tok_off, tr_sha, off_sha, B, caps, direct_idx, threads, log):
    t = {}
    t0 = time.time()
    off = oracle.block_offsets(req_tok_off, B)
    prev, nxt = oracle.reuse(ids, D)
    t["reuse"] = time.time() - t0
    t0 = time.time()
    sd = oracle.sd_fenwick(prev)
    t["sd_fenwick"] = time.time() - t0
    out = {"N": int(ids.size), "D": int(D), "B": B, "tokens_sha256": tr_sha, "req_tok_off_sha256": off_sha,
           "ids_sha256": sha(ids), "prev_sha256": sha(prev), "next_sha256": sha(nxt), "dist_sha256": sha(sd),
           "caps": [int(c) for c in caps]}
    del prev, nxt
    gc.collect()
    t0 = time.time()
    hits, saved = oracle.curves_from_dist(sd, off, B, caps)
    t["curves_from_dist"] = time.time() - t0
    out["hits"] = hits
    out["saved"] = [str(s) for s in saved]
    del sd
    gc.collect()
    t0 = time.time()
    dcaps = caps[np.asarray(direct_idx)]
    h, s, total = oracle.lru_curves(ids, off, B, dcaps, threads=threads)
    t["lru_direct"] = time.time() - t0
    out["total_cost"] = str(total)
    out["direct"] = {"index": [int(i) for i in direct_idx], "hits": h, "saved": [str(x) for x in s]}
    # the two routes must agree at the directly simulated points (inclusion)
    assert [hits[i] for i in direct_idx] == h and [saved[i] for i in direct_idx] == s
    out["oracle_seconds"] = {k: round(v, 1) for k, v in t.items()}
    log(f"  B={B}: N={ids.size} D={D} {out['oracle_seconds']} peak {peak_gb():.1f} GB")
    return out



def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--only", choices=["agentic", "mixed"], default=None)
    ap.add_argument("--threads", type=int, default=os.cpu_count() or 1)
    args = ap.parse_args()
    data = {}
    if os.path.exists(OUT):
        with open(OUT) as f:
            data = json.load(f)

    def log(msg):
        print(msg, flush=True)

    def save():
        data["_about"] = ("Oracle results on the full-size agentic (seed 2) and mixed 24-hour (seed 3) traces; "
                          "written by tests/golden/make_big_goldens.py, which calls only oracle/ and tracegen/.")
        with open(OUT, "w") as f:
            json.dump(data, f, indent=1, sort_keys=True)
            f.write("\n")

    if args.only in (None, "agentic"):
        t0 = time.time()
        tr = tracegen.make(2)
        tr_sha, off_sha = sha(tr.tokens), sha(tr.req_tok_off)
        log(f"agentic: {tr.n_tok} tokens, {tr.n_req} requests, generated in {time.time() - t0:.1f} s")
        d16 = None
        for B in (16, 32, 64, 256):
            t0 = time.time()
            ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, B)
            tid = time.time() - t0
            if B == 16:
                d16 = D
            caps = token_grid(d16, B)
            G = len(caps)
            e = entry(ids, D, tr.req_tok_off, tr_sha, off_sha, B, caps, [G // 8, 3 * G // 8, 5 * G // 8, 7 * G // 8], args.threads,
                      log)
            e["oracle_seconds"]["block_ids"] = round(tid, 1)
            e["workload"] = 2
            e["grid"] = "16 x capacity_grid(round(0.001 D16), D16, 128) tokens, as blocks of B (D16 = D at B = 16)"
            data[f"agentic_B{B}"] = e
            del ids
            gc.collect()
            save()
        del tr
        gc.collect()

    if args.only in (None, "mixed"):
        t0 = time.time()
        tr = tracegen.make(3)
        tr_sha, off_sha = sha(tr.tokens), sha(tr.req_tok_off)
        log(f"mixed: {tr.n_tok} tokens, {tr.n_req} requests, generated in {time.time() - t0:.1f} s")
        t0 = time.time()
        ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
        tid = time.time() - t0
        log(f"  ids in {tid:.1f} s, peak {peak_gb():.1f} GB")
        tr.tokens = None
        gc.collect()
        caps = tracegen.workload_grid(3, D)
        # direct simulation at eight grid points whose LRU state fits in memory together
        e = entry(ids, D, tr.req_tok_off, tr_sha, off_sha, 16, caps, [0, 16, 32, 48, 64, 80, 96, 104], args.threads, log)
        e["oracle_seconds"]["block_ids"] = round(tid, 1)
        e["workload"] = 3
        e["grid"] = "capacity_grid(round(0.001 D), D, 128)"
        data["mixed_B16"] = e
        save()


if __name__ == "__main__":
    main()
