"""CPU ORACLE — test infrastructure only.

A plain, slow, obviously correct CPU implementation of the prefix-cache curve
computation (``oracle.cpp``), wrapped for numpy.  Only ``tests/``, the smoke
check in ``__graft_entry__`` and ``bench.py``'s CPU-baseline leg may import
this package; the product path (``paper_2609_28870_gb300``) never does.

Functions and the passages they restate:

* ``block_offsets``, ``block_ids`` — Sec. 2.2: 16-token KV blocks, reusable iff
  the whole preceding sequence matches; exact trie identity, ids numbered by
  first occurrence.
* ``reuse`` — previous / next access of each block (Belady's next use, Sec. 3.2).
* ``sd_mattson``, ``sd_fenwick`` — LRU stack distance (App. B), by Mattson's
  move-to-front stack and by Bennett-Kruskal counting.
* ``lru_curves`` — direct LRU simulation per capacity (Sec. 3.1-3.2) with
  prefix-contiguous hits (Sec. 2.2) and compute saved (Sec. 5.2, App. C).
* ``curves_from_dist`` — the same curves from stack distances by Mattson
  inclusion (App. B).
* ``belady_curves`` — Belady's offline optimum (Sec. 3.2): direct MIN
  simulation per capacity, same prefix rule and costs.
* ``session_lru_curves`` — session-level LRU eviction (Sec. 5.3): direct
  simulation per capacity, evicting the least recent session's blocks whole.
* ``lru_curves_variant``, ``sd_variant`` — Sec. 3.1: leaf-first touch order
  and whole-request residency (every block looked up at the request's
  arrival), by direct LRU per capacity, Fenwick counting and Mattson's list.
* ``trace_stats`` — Sec. 4.1-4.3 and App. B: per-category block counts,
  frequency, lifetime and reuse-interval histograms, session lengths and
  durations, and reuses reachable within each capacity.
* ``prefix_hash`` — the polynomial prefix key the GPU path writes,
  sum_t (tok_t + 1) u^(t+1) mod 2^61 - 1 at two seeded bases, token by token.
* ``run`` — all of the above on one trace.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.cpp")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

NONE = 0xFFFFFFFF

# Cost-model kinds (Sec. 5.2 and App. C)
COST_UNIFORM, COST_MEASURED, COST_LINEAR = 0, 1, 2
# Per-token constants of the measured-shape model: F_lin = 2 * 3.3e9 FLOPs per
# token for the active parameters; F_attn = 4 * 48 layers * 32 heads * 128 dims
# per attended position.
F_LIN = 6_600_000_000
F_ATTN = 4 * 48 * 32 * 128


def build(force: bool = False) -> str:
    """Compile ``oracle.cpp`` into ``oracle/_build/liboracle.so``."""
    with _lock:
        if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
            return _LIB
        os.makedirs(_BUILD, exist_ok=True)
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread", _SRC, "-o", tmp], check=True)
        os.replace(tmp, _LIB)
        return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        vp, u32, u64, i32 = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int
        lib.orc_block_offsets.restype = u64
        lib.orc_block_offsets.argtypes = [vp, u32, u32, vp]
        lib.orc_block_ids.restype = u64
        lib.orc_block_ids.argtypes = [vp, vp, u32, u32, vp]
        lib.orc_reuse.argtypes = [vp, u64, u64, vp, vp]
        lib.orc_sd_mattson.argtypes = [vp, u64, vp]
        lib.orc_sd_fenwick.argtypes = [vp, u64, vp]
        lib.orc_lru_curves.restype = i32
        lib.orc_lru_curves.argtypes = [vp, vp, u32, u32, i32, u64, u64, vp, u32, i32, vp, vp, vp, vp, vp]
        lib.orc_prefix_hash.argtypes = [vp, vp, u32, u32, u64, vp]
        lib.orc_session_lru_curves.restype = i32
        lib.orc_session_lru_curves.argtypes = [vp, vp, vp, u32, u32, u32, i32, u64, u64, vp, u32, i32, vp, vp, vp]
        lib.orc_belady_curves.restype = i32
        lib.orc_belady_curves.argtypes = [vp, vp, u32, u32, i32, u64, u64, vp, u32, i32, vp, vp, vp, vp]
        lib.orc_curves_from_dist.restype = i32
        lib.orc_curves_from_dist.argtypes = [vp, vp, u32, u32, i32, u64, u64, vp, u32, vp, vp, vp]
        lib.orc_lru_curves_variant.restype = i32
        lib.orc_lru_curves_variant.argtypes = [vp, vp, u32, u32, i32, u64, u64, vp, u32, i32, i32, i32, vp, vp, vp]
        lib.orc_sd_variant.restype = i32
        lib.orc_sd_variant.argtypes = [vp, u64, vp, u32, i32, i32, vp]
        lib.orc_sd_variant_mattson.restype = i32
        lib.orc_sd_variant_mattson.argtypes = [vp, vp, u32, i32, i32, vp]
        lib.orc_trace_stats.restype = i32
        lib.orc_trace_stats.argtypes = [vp, u64, u64, vp, vp, vp, u32, u64, vp, vp, u32] + [vp] * 13
        _lib = lib
    return _lib


def _p(a):
    return a.ctypes.data


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def block_offsets(req_tok_off, B: int) -> np.ndarray:
    off = _c(req_tok_off, np.uint64)
    out = np.empty(off.shape[0], dtype=np.uint64)
    _load().orc_block_offsets(_p(off), off.shape[0] - 1, int(B), _p(out))
    return out


def block_ids(tokens, req_tok_off, B: int):
    """(ids uint32[N], D) with exact prefix identity."""
    tok, off = _c(tokens, np.uint32), _c(req_tok_off, np.uint64)
    n = int(block_offsets(off, B)[-1])
    ids = np.empty(n, dtype=np.uint32)
    d = _load().orc_block_ids(_p(tok), _p(off), off.shape[0] - 1, int(B), _p(ids))
    return ids, int(d)


def reuse(ids, n_distinct: int):
    ids = _c(ids, np.uint32)
    prev = np.empty_like(ids)
    nxt = np.empty_like(ids)
    _load().orc_reuse(_p(ids), ids.shape[0], int(n_distinct), _p(prev), _p(nxt))
    return prev, nxt


def sd_mattson(ids) -> np.ndarray:
    ids = _c(ids, np.uint32)
    sd = np.empty_like(ids)
    _load().orc_sd_mattson(_p(ids), ids.shape[0], _p(sd))
    return sd


def sd_fenwick(prev) -> np.ndarray:
    prev = _c(prev, np.uint32)
    sd = np.empty_like(prev)
    _load().orc_sd_fenwick(_p(prev), prev.shape[0], _p(sd))
    return sd


def lru_curves(ids, req_blk_off, B: int, caps, kind: int = COST_MEASURED, f_lin: int = F_LIN,
               f_attn: int = F_ATTN, threads: int | None = None):
    """Direct LRU simulation at each capacity.  Returns (hits list[int],
    saved list[int] (exact, from 128-bit sums), total_cost int)."""
    ids, bo, caps = _c(ids, np.uint32), _c(req_blk_off, np.uint64), _c(caps, np.uint64)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    slo = np.zeros(G, dtype=np.uint64)
    shi = np.zeros(G, dtype=np.uint64)
    tlo = np.zeros(1, dtype=np.uint64)
    thi = np.zeros(1, dtype=np.uint64)
    nthreads = threads or max(1, min(G, os.cpu_count() or 1))
    rc = _load().orc_lru_curves(_p(ids), _p(bo), bo.shape[0] - 1, int(B), int(kind), int(f_lin), int(f_attn),
                                _p(caps), G, nthreads, _p(hits), _p(slo), _p(shi), _p(tlo), _p(thi))
    if rc != 0:
        raise ValueError("bad capacity grid (capacities must be >= 1)")
    saved = [int(h) << 64 | int(l) for l, h in zip(slo, shi)]
    return [int(h) for h in hits], saved, int(thi[0]) << 64 | int(tlo[0])


def session_lru_curves(ids, req_blk_off, req_session, n_session: int, B: int, caps, kind: int = COST_MEASURED,
                       f_lin: int = F_LIN, f_attn: int = F_ATTN, threads: int | None = None):
    """Session-level LRU (Sec. 5.3) simulated directly at each capacity: a
    block belongs to the session that brought it in; the least recently
    touched other session is evicted whole while more than C blocks are
    resident; a session alone above C keeps only the block just brought in.
    Prefix rule and costs as lru_curves.  Returns (hits, saved)."""
    ids, bo, caps = _c(ids, np.uint32), _c(req_blk_off, np.uint64), _c(caps, np.uint64)
    ses = _c(req_session, np.uint32)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    slo = np.zeros(G, dtype=np.uint64)
    shi = np.zeros(G, dtype=np.uint64)
    nthreads = threads or max(1, min(G, os.cpu_count() or 1))
    rc = _load().orc_session_lru_curves(_p(ids), _p(bo), _p(ses), bo.shape[0] - 1, int(n_session), int(B), int(kind),
                                        int(f_lin), int(f_attn), _p(caps), G, nthreads, _p(hits), _p(slo), _p(shi))
    if rc != 0:
        raise ValueError("bad capacity grid or session label")
    return [int(h) for h in hits], [int(h) << 64 | int(l) for l, h in zip(slo, shi)]


def belady_curves(ids, req_blk_off, B: int, caps, kind: int = COST_MEASURED, f_lin: int = F_LIN,
                  f_attn: int = F_ATTN, threads: int | None = None):
    """Belady's MIN simulated directly at each capacity (evict the resident
    block, other than the one just brought in, whose next access is farthest;
    every access admitted), with the prefix rule.  Returns (hits list[int],
    saved list[int], raw_hits list[int]); raw hits ignore the prefix rule."""
    ids, bo, caps = _c(ids, np.uint32), _c(req_blk_off, np.uint64), _c(caps, np.uint64)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    raw = np.zeros(G, dtype=np.uint64)
    slo = np.zeros(G, dtype=np.uint64)
    shi = np.zeros(G, dtype=np.uint64)
    nthreads = threads or max(1, min(G, os.cpu_count() or 1))
    rc = _load().orc_belady_curves(_p(ids), _p(bo), bo.shape[0] - 1, int(B), int(kind), int(f_lin), int(f_attn),
                                   _p(caps), G, nthreads, _p(hits), _p(slo), _p(shi), _p(raw))
    if rc != 0:
        raise ValueError("bad capacity grid (capacities must be >= 1)")
    return [int(h) for h in hits], [int(h) << 64 | int(l) for l, h in zip(slo, shi)], [int(x) for x in raw]


def curves_from_dist(sd, req_blk_off, B: int, caps, kind: int = COST_MEASURED, f_lin: int = F_LIN,
                     f_attn: int = F_ATTN):
    """Hits and compute saved per capacity from stack distances by Mattson
    inclusion (running maximum per request, root-first).  Returns (hits
    list[int], saved list[int]); caps strictly ascending."""
    sd, bo, caps = _c(sd, np.uint32), _c(req_blk_off, np.uint64), _c(caps, np.uint64)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    slo = np.zeros(G, dtype=np.uint64)
    shi = np.zeros(G, dtype=np.uint64)
    rc = _load().orc_curves_from_dist(_p(sd), _p(bo), bo.shape[0] - 1, int(B), int(kind), int(f_lin), int(f_attn),
                                      _p(caps), G, _p(hits), _p(slo), _p(shi))
    if rc != 0:
        raise ValueError("bad capacity grid (capacities must be >= 1 and strictly ascending)")
    return [int(h) for h in hits], [int(h) << 64 | int(l) for l, h in zip(slo, shi)]


def prefix_hash(tokens, req_tok_off, B: int, seed: int) -> np.ndarray:
    """Keys uint64[N, 2]: the polynomial prefix hash with the two seeded bases."""
    tok, off = _c(tokens, np.uint32), _c(req_tok_off, np.uint64)
    n = int(block_offsets(off, B)[-1])
    keys = np.empty((n, 2), dtype=np.uint64)
    _load().orc_prefix_hash(_p(tok), _p(off), off.shape[0] - 1, int(B), int(seed) & (2**64 - 1), _p(keys))
    return keys


# Semantics variants (Sec. 3.1): the order a request's blocks are touched in,
# and whether they are looked up one by one or all at the request's arrival.
ROOT_FIRST, LEAF_FIRST = 0, 1
RES_BLOCK, RES_REQUEST = 0, 1


def lru_curves_variant(ids, req_blk_off, B: int, caps, order: int, residency: int, kind: int = COST_MEASURED,
                       f_lin: int = F_LIN, f_attn: int = F_ATTN, threads: int | None = None):
    """Direct LRU simulation per capacity under a touch order and a
    residency rule.  Returns (hits list[int], saved list[int])."""
    ids, bo, caps = _c(ids, np.uint32), _c(req_blk_off, np.uint64), _c(caps, np.uint64)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    slo = np.zeros(G, dtype=np.uint64)
    shi = np.zeros(G, dtype=np.uint64)
    nthreads = threads or max(1, min(G, os.cpu_count() or 1))
    rc = _load().orc_lru_curves_variant(_p(ids), _p(bo), bo.shape[0] - 1, int(B), int(kind), int(f_lin), int(f_attn),
                                        _p(caps), G, int(order), int(residency), nthreads, _p(hits), _p(slo), _p(shi))
    if rc != 0:
        raise ValueError("bad capacity grid or variant")
    return [int(h) for h in hits], [int(h) << 64 | int(l) for l, h in zip(slo, shi)]


def sd_variant(ids, n_distinct: int, req_blk_off, order: int, residency: int, mattson: bool = False) -> np.ndarray:
    """Stack distance of every access under a variant, in depth order."""
    ids, bo = _c(ids, np.uint32), _c(req_blk_off, np.uint64)
    sd = np.empty_like(ids)
    if mattson:
        rc = _load().orc_sd_variant_mattson(_p(ids), _p(bo), bo.shape[0] - 1, int(order), int(residency), _p(sd))
    else:
        rc = _load().orc_sd_variant(_p(ids), int(n_distinct), _p(bo), bo.shape[0] - 1, int(order), int(residency),
                                    _p(sd))
    if rc != 0:
        raise ValueError("bad variant")
    return sd


# Shapes of the trace statistics: category-major histograms have 3 rows
# (0 shared across sessions, 1 session history, 2 single-turn); log2 bins are
# the bit length of the value (65 bins); freq has 256 exact bins with the
# blocks used 256 times or more in bin 0.
STAT_SHAPES = dict(blocks=(3,), accesses=(3,), freq=(3, 256), freq_log2=(3, 65), reuse_us=(3, 65),
                   lifetime_us=(3, 65), reuse_by_freq=(65, 65), lifetime_by_freq=(65, 65), dist_log2=(65,),
                   sess_requests=(65,), sess_duration_us=(65,))
STAT_SCALARS = ("n_access", "n_distinct", "n_reuse", "n_sessions", "n_multi_sessions")


def trace_stats(ids, n_distinct: int, req_blk_off, req_ts_us, req_session, n_session: int, dist=None,
                caps=None) -> dict:
    """Trace statistics of Sec. 4.1-4.3 and App. B (see orc_trace_stats):
    uint64 histograms named as in STAT_SHAPES, the STAT_SCALARS, and
    ``reach`` (reuses with stack distance <= caps[g]) when dist is given."""
    ids, bo = _c(ids, np.uint32), _c(req_blk_off, np.uint64)
    ts, ses = _c(req_ts_us, np.int64), _c(req_session, np.uint64)
    caps = _c([] if caps is None else caps, np.uint64)
    out = {k: np.zeros(v, dtype=np.uint64) for k, v in STAT_SHAPES.items()}
    reach = np.zeros(max(caps.shape[0], 1), dtype=np.uint64)
    scal = np.zeros(len(STAT_SCALARS), dtype=np.uint64)
    dptr = None
    if dist is not None:
        dist = _c(dist, np.uint32)
        dptr = _p(dist)
    rc = _load().orc_trace_stats(_p(ids), ids.shape[0], int(n_distinct), _p(bo), _p(ts), _p(ses),
                                 bo.shape[0] - 1, int(n_session), dptr, _p(caps), caps.shape[0],
                                 *[_p(out[k]) for k in list(STAT_SHAPES)[:9]], _p(reach),
                                 _p(out["sess_requests"]), _p(out["sess_duration_us"]), _p(scal))
    if rc == 1:
        raise ValueError("malformed trace (ids, sessions or offsets)")
    if rc == 2:
        raise ValueError("request timestamps decrease")
    out.update({k: int(v) for k, v in zip(STAT_SCALARS, scal)})
    if dist is not None:
        out["reach"] = reach[: caps.shape[0]]
    return out


def run(tokens, req_tok_off, B: int, caps, kind: int = COST_MEASURED, f_lin: int = F_LIN, f_attn: int = F_ATTN,
        threads: int | None = None, mattson: bool = False) -> dict:
    """Every oracle stage on one trace."""
    off = block_offsets(req_tok_off, B)
    ids, D = block_ids(tokens, req_tok_off, B)
    prev, nxt = reuse(ids, D)
    sd = sd_fenwick(prev)
    out = dict(req_blk_off=off, ids=ids, n_access=int(ids.shape[0]), n_distinct=D, prev=prev, next=nxt, sd=sd)
    if mattson:
        out["sd_mattson"] = sd_mattson(ids)
    hits, saved, total = lru_curves(ids, off, B, caps, kind, f_lin, f_attn, threads)
    out.update(hits=hits, saved=saved, total_cost=total)
    return out
