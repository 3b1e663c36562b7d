"""Seeded synthetic request traces shaped like the paper's workloads.

This module draws inputs only; it contains none of the method's arithmetic.
Both the CPU oracle (``oracle/``) and the GPU path read the arrays it returns.

    tr = tracegen.make(1)                  # conversational chat workload, seed 1
    tr.tokens, tr.req_tok_off, tr.req_ts_us, tr.req_session   (numpy arrays)

Workloads (the session count is the scale knob; every other parameter follows
the stated distribution):

    0  tiny conversational trace   444 sessions  -> ~2,000 requests
    1  conversational chat trace   5,600 sessions -> ~150M tokens
    2  agentic coding trace        560 sessions  -> ~2.1B tokens, 131,072 cap
    3  mixed 24 h trace            chat + agentic halves, diurnal arrivals

The generator is C++ (``tracegen.cpp``), built on first use with g++ and
``-ffp-contract=off`` so that x86-64 and aarch64 hosts emit identical traces.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tracegen.cpp")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libtracegen.so")
_lock = threading.Lock()
_lib = None

WORKLOADS = {
    0: "tiny conversational trace (seed 0, 444 sessions, B=16, 16-point grid)",
    1: "conversational chat trace (seed 1, 5,600 sessions, ~150M tokens, B=16, 64-point grid)",
    2: "agentic coding trace (seed 2, 560 sessions, ~2.1B tokens, 131,072-token cap, B=16)",
    3: "mixed 24 h trace (seed 3, chat + agentic halves, diurnal arrivals, ~10B tokens)",
}
DEFAULT_SEED = {0: 0, 1: 1, 2: 2, 3: 3}


def build(force: bool = False) -> str:
    """Compile the generator into ``tracegen/_build/libtracegen.so``."""
    with _lock:
        if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
            return _LIB
        os.makedirs(_BUILD, exist_ok=True)
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
               "-pthread", _SRC, "-o", tmp]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
        return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        vp, u64 = ctypes.c_void_p, ctypes.c_uint64
        lib.tg_make.restype = vp
        lib.tg_make.argtypes = [ctypes.c_int, u64, ctypes.c_int64, ctypes.c_int64]
        lib.tg_sizes.argtypes = [vp] + [ctypes.POINTER(u64)] * 3
        lib.tg_offsets.argtypes = [vp, u64, vp, vp, vp]
        lib.tg_fill_tokens.argtypes = [vp, u64, vp, vp, ctypes.c_int]
        lib.tg_free.argtypes = [vp]
        for name in ("tg_det_log", "tg_det_exp", "tg_det_cos"):
            getattr(lib, name).restype = ctypes.c_double
            getattr(lib, name).argtypes = [ctypes.c_double]
        lib.tg_sm64_at.restype = u64
        lib.tg_sm64_at.argtypes = [u64, u64]
        _lib = lib
    return _lib


@dataclass
class Trace:
    tokens: np.ndarray       # uint32[T]
    req_tok_off: np.ndarray  # uint64[R+1]
    req_ts_us: np.ndarray    # int64[R]
    req_session: np.ndarray  # uint64[R]
    n_sessions: int = 0
    workload: int = -1
    seed: int = 0

    @property
    def n_req(self) -> int:
        return int(self.req_ts_us.shape[0])

    @property
    def n_tok(self) -> int:
        return int(self.req_tok_off[-1])

    def head(self, n_req: int) -> "Trace":
        """The first ``n_req`` requests in trace order (a valid, shorter trace)."""
        n_req = min(n_req, self.n_req)
        end = int(self.req_tok_off[n_req])
        return Trace(self.tokens[:end], self.req_tok_off[: n_req + 1], self.req_ts_us[:n_req],
                     self.req_session[:n_req], self.n_sessions, self.workload, self.seed)


def from_lists(requests, ts=None, sessions=None) -> Trace:
    """A hand-written trace: ``requests`` is a list of token lists in trace order."""
    lens = [len(r) for r in requests]
    off = np.zeros(len(requests) + 1, dtype=np.uint64)
    off[1:] = np.cumsum(np.asarray(lens, dtype=np.uint64)) if requests else []
    tokens = np.asarray([t for r in requests for t in r], dtype=np.uint32)
    R = len(requests)
    ts_arr = np.arange(R, dtype=np.int64) if ts is None else np.asarray(ts, dtype=np.int64)
    ses = np.zeros(R, dtype=np.uint64) if sessions is None else np.asarray(sessions, dtype=np.uint64)
    return Trace(tokens, off, ts_arr, ses, int(len(set(ses.tolist()))) if R else 0)


def make(workload: int, seed: int | None = None, sessions: int = 0, sessions_b: int = 0,
         max_requests: int | None = None, threads: int | None = None, token_buffer=None) -> Trace:
    """Generate workload ``workload`` (0-3).

    ``sessions``/``sessions_b`` override the session counts (``sessions_b`` is
    the agentic half of workload 3).  ``max_requests`` keeps a prefix in trace
    order.  ``token_buffer`` may be a preallocated uint32 numpy array (for
    example a view of pinned host memory) at least as long as the trace."""
    lib = _load()
    if seed is None:
        seed = DEFAULT_SEED[workload]
    h = lib.tg_make(int(workload), ctypes.c_uint64(seed), int(sessions), int(sessions_b))
    if not h:
        raise ValueError(f"unknown workload {workload}")
    try:
        n_req, n_tok, n_ses = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
        lib.tg_sizes(h, ctypes.byref(n_req), ctypes.byref(n_tok), ctypes.byref(n_ses))
        R = n_req.value if max_requests is None else min(n_req.value, int(max_requests))
        off = np.empty(R + 1, dtype=np.uint64)
        ts = np.empty(R, dtype=np.int64)
        ses = np.empty(R, dtype=np.uint64)
        lib.tg_offsets(h, R, off.ctypes.data, ts.ctypes.data, ses.ctypes.data)
        total = int(off[-1])
        if token_buffer is None:
            tokens = np.empty(total, dtype=np.uint32)
        else:
            if token_buffer.dtype != np.uint32 or token_buffer.shape[0] < total:
                raise ValueError("token_buffer is not uint32 or too short")
            tokens = token_buffer[:total]
        nthreads = threads or max(1, min(32, os.cpu_count() or 1))
        lib.tg_fill_tokens(h, R, off.ctypes.data, tokens.ctypes.data, nthreads)
        return Trace(tokens, off, ts, ses, int(n_ses.value), int(workload), int(seed))
    finally:
        lib.tg_free(h)


def sizes(workload: int, seed: int | None = None, sessions: int = 0, sessions_b: int = 0):
    """(requests, tokens, sessions) of a workload without materialising tokens."""
    lib = _load()
    if seed is None:
        seed = DEFAULT_SEED[workload]
    h = lib.tg_make(int(workload), ctypes.c_uint64(seed), int(sessions), int(sessions_b))
    try:
        n_req, n_tok, n_ses = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
        lib.tg_sizes(h, ctypes.byref(n_req), ctypes.byref(n_tok), ctypes.byref(n_ses))
        return int(n_req.value), int(n_tok.value), int(n_ses.value)
    finally:
        lib.tg_free(h)


def capacity_grid(c_lo: int, c_hi: int, G: int) -> np.ndarray:
    """Log-spaced capacity grid in blocks (an input to both sides, as integers).

    c_g = round(c_lo * (c_hi / c_lo) ** (g / (G - 1))); a point that would not
    exceed its predecessor becomes predecessor + 1; the last point is c_hi
    whenever that keeps the grid strictly ascending."""
    c_lo, c_hi = max(1, int(c_lo)), max(1, int(c_hi))
    c_hi = max(c_hi, c_lo)
    out = []
    for g in range(G):
        v = c_lo if G == 1 else int(round(c_lo * (c_hi / c_lo) ** (g / (G - 1))))
        if out and v <= out[-1]:
            v = out[-1] + 1
        out.append(v)
    if G > 1 and out[-2] < c_hi:
        out[-1] = c_hi
    return np.asarray(out, dtype=np.uint64)


# Capacity grid of each workload as (c_lo, c_hi, G) given D distinct blocks.
def workload_grid(workload: int, n_distinct: int) -> np.ndarray:
    if workload == 0:
        return capacity_grid(64, n_distinct, 16)
    if workload in (1, 2):
        return capacity_grid(64, n_distinct, 64)
    return capacity_grid(max(1, round(0.001 * n_distinct)), n_distinct, 128)


def tiny(seed: int, n_sessions: int = 6, max_turns: int = 5, vocab: int = 3, sys_pool: int = 2,
         max_seg: int = 7, truncate_prob: float = 0.25) -> Trace:
    """A small random trace with the structure of the large workloads: sessions
    that share system prompts and append turns, interleaved in time, with
    occasional truncation (a dropped middle turn) and requests shorter than a
    block.  A tiny vocabulary makes equal block contents under different
    prefixes common.  Pure numpy; for unit tests and brute-force checks."""
    rng = np.random.default_rng(seed)
    sys_prompts = [list(rng.integers(0, vocab, rng.integers(0, max_seg + 1))) for _ in range(sys_pool)]
    events = []
    for s in range(n_sessions):
        t = float(rng.uniform(0, 100))
        ctx = [list(sys_prompts[rng.integers(0, sys_pool)])]
        for turn in range(int(rng.integers(1, max_turns + 1))):
            ctx.append(list(rng.integers(0, vocab, rng.integers(0, max_seg + 1))))
            if len(ctx) > 2 and rng.random() < truncate_prob:
                del ctx[1]
            events.append((t, s, turn, [int(x) for seg in ctx for x in seg]))
            t += float(rng.uniform(0.5, 20))
    events.sort(key=lambda e: (e[0], e[1], e[2]))
    ts = [int(e[0] * 1e6) for e in events]
    return from_lists([e[3] for e in events], ts=ts, sessions=[e[1] for e in events])
