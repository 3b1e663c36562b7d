"""ptc — prefix-cache curves on one GPU (GB300, sm_103a).

A thin binding over the C-ABI library ``libptc.so`` (declared in
``include/ptc.h``).  Each function marshals arguments and calls the C entry
point of the same name; every step of the computation runs in the library's
CUDA kernels.  PyTorch provides device memory and the current CUDA stream.

    keys, req_blk_off, n = ptc_hash_blocks(tokens, req_tok_off, req_ts_us, 16, seed)
    ids, d               = ptc_assign_ids(keys)
    prev, nxt            = ptc_reuse_indices(ids, d)
    dist                 = ptc_stack_distance(prev)
    curves               = ptc_curves(dist, req_blk_off, 16, caps, PTC_COST_MEASURED)

Arrays are torch CUDA tensors.  Unsigned 32/64-bit arrays travel as int32 /
int64 tensors holding the same bits (``u32()`` / ``u64()`` give numpy views).
There is no CPU fallback: without the built library every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

from . import build as _build

PTC_NONE = 0xFFFFFFFF
PTC_COST_UNIFORM, PTC_COST_MEASURED, PTC_COST_LINEAR = 0, 1, 2
PTC_SD_AUTO, PTC_SD_POINTS, PTC_SD_RUNS = 0, 1, 2
PTC_REUSE_AUTO, PTC_REUSE_SORT, PTC_REUSE_RUNS = 0, 1, 2
PTC_IDS_AUTO, PTC_IDS_TABLE, PTC_IDS_PARTITIONED = 0, 1, 2
PTC_TOUCH_ROOT_FIRST, PTC_TOUCH_LEAF_FIRST = 0, 1
PTC_RESIDENCY_BLOCK, PTC_RESIDENCY_REQUEST = 0, 1
F_LIN = 6_600_000_000          # 2 x 3.3e9 active parameters, FLOPs per token
F_ATTN = 4 * 48 * 32 * 128     # per attended position: 4 x layers x heads x head_dim
MAX_CAPACITIES = 1024
MAX_BLOCK_SIZE = 512

_lock = threading.Lock()
_lib = None

STATUS = {
    0: "PTC_OK", 1: "PTC_ERR_INVALID_ARG", 2: "PTC_ERR_UNSORTED", 3: "PTC_ERR_OVERFLOW",
    4: "PTC_ERR_WORKSPACE", 5: "PTC_ERR_CUDA", 6: "PTC_ERR_TIMEOUT", 7: "PTC_ERR_HASH_COLLISION",
    8: "PTC_ERR_NOT_IMPLEMENTED", 9: "PTC_ERR_BOUNDS",
}


class PtcError(RuntimeError):
    def __init__(self, call: str, status: int):
        self.status = status
        self.name = STATUS.get(status, str(status))
        super().__init__(f"{call}: {self.name} ({lib().ptc_strerror(status).decode()})")


class CostModel(ctypes.Structure):
    _fields_ = [("f_lin", ctypes.c_uint64), ("f_attn", ctypes.c_uint64), ("kind", ctypes.c_int32)]


class U128(ctypes.Structure):
    _fields_ = [("lo", ctypes.c_uint64), ("hi", ctypes.c_uint64)]


_lib_path = None


def library_path() -> str:
    return _lib_path or _build.LIB


def use_checked_build() -> str:
    """Load the checked build (``build(checked=True)``: every index read from
    data is checked, PTC_ERR_BOUNDS on a miss) instead of the normal one.  Must
    come before the first call into the library in this process."""
    global _lib_path
    if _lib is not None:
        raise RuntimeError("the library is already loaded in this process")
    _lib_path = _build.LIB_CHECKED
    return _lib_path


def lib():
    """The loaded ``libptc.so``.  Raises if it has not been built."""
    global _lib
    if _lib is None:
        with _lock:
            if _lib is None:
                path = library_path()
                if not os.path.exists(path):
                    raise RuntimeError(f"libptc.so is not built ({path}); run "
                                       "`python -c 'import __graft_entry__ as g; g.build()'`")
                L = ctypes.CDLL(path)
                vp, u32, u64, i64, sz = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int64, ctypes.c_size_t
                st = ctypes.c_int
                L.ptc_strerror.restype = ctypes.c_char_p
                L.ptc_strerror.argtypes = [st]
                L.ptc_version.restype = ctypes.c_char_p
                L.ptc_version.argtypes = []
                L.ptc_hash_blocks_workspace_bytes.restype = sz
                L.ptc_hash_blocks_workspace_bytes.argtypes = [u32, u64, u32]
                L.ptc_hash_blocks.restype = st
                L.ptc_hash_blocks.argtypes = [vp, u64, vp, vp, u32, u32, u64, vp, u64, vp,
                                              ctypes.POINTER(u64), vp, sz, vp]
                L.ptc_assign_ids_workspace_bytes.restype = sz
                L.ptc_assign_ids_workspace_bytes.argtypes = [u64]
                L.ptc_assign_ids.restype = st
                L.ptc_assign_ids.argtypes = [vp, u64, vp, ctypes.POINTER(u64), vp, sz, vp]
                L.ptc_verify_ids_workspace_bytes.restype = sz
                L.ptc_verify_ids_workspace_bytes.argtypes = [u64, u64]
                L.ptc_verify_ids.restype = st
                L.ptc_verify_ids.argtypes = [vp, u64, vp, vp, u32, u32, vp, u64, u64, vp, sz, vp]
                L.ptc_reuse_indices_workspace_bytes.restype = sz
                L.ptc_reuse_indices_workspace_bytes.argtypes = [u64, u64]
                L.ptc_reuse_indices.restype = st
                L.ptc_reuse_indices.argtypes = [vp, u64, u64, vp, vp, vp, sz, vp]
                L.ptc_stack_distance_workspace_bytes.restype = sz
                L.ptc_stack_distance_workspace_bytes.argtypes = [u64]
                L.ptc_stack_distance.restype = st
                L.ptc_stack_distance.argtypes = [vp, u64, vp, vp, sz, vp]
                L.ptc_reuse_indices_ex_workspace_bytes.restype = sz
                L.ptc_reuse_indices_ex_workspace_bytes.argtypes = [u64, u64, ctypes.c_int]
                L.ptc_reuse_indices_ex.restype = st
                L.ptc_reuse_indices_ex.argtypes = [vp, u64, u64, vp, vp, ctypes.c_int, vp, sz, vp]
                L.ptc_stack_distance_ex_workspace_bytes.restype = sz
                L.ptc_stack_distance_ex_workspace_bytes.argtypes = [u64, ctypes.c_int]
                L.ptc_stack_distance_ex.restype = st
                L.ptc_stack_distance_ex.argtypes = [vp, u64, vp, ctypes.c_int, vp, sz, vp]
                L.ptc_curves_workspace_bytes.restype = sz
                L.ptc_curves_workspace_bytes.argtypes = [u64, u32, u32]
                L.ptc_curves.restype = st
                L.ptc_curves.argtypes = [vp, u64, vp, u32, u32, ctypes.POINTER(CostModel), vp, u32, vp, vp,
                                         ctypes.POINTER(U128), vp, sz, vp]
                L.ptc_pipeline_workspace_bytes.restype = sz
                L.ptc_pipeline_workspace_bytes.argtypes = [u32, u64, u32, u32]
                L.ptc_probe_random_rmw.restype = st
                L.ptc_probe_random_rmw.argtypes = [vp, u64, u64, u64, vp, vp]
                L.ptc_pipeline.restype = st
                L.ptc_pipeline.argtypes = [vp, u64, vp, vp, vp, u32, u32, u32, u64, ctypes.POINTER(CostModel), vp, u32,
                                           vp, vp, vp, vp, vp, vp, ctypes.POINTER(u64), ctypes.POINTER(u64), vp, vp,
                                           ctypes.POINTER(U128), vp, sz, vp]
                L.ptc_pipeline_host_workspace_bytes.restype = sz
                L.ptc_pipeline_host_workspace_bytes.argtypes = [u32, u64, u32, u32]
                L.ptc_pipeline_host.restype = st
                L.ptc_pipeline_host.argtypes = [vp, u64, vp, vp, vp, u32, u32, u32, u64, ctypes.POINTER(CostModel),
                                                vp, u32,
                                                ctypes.POINTER(u64), ctypes.POINTER(u64), vp, vp, ctypes.POINTER(U128),
                                                vp, sz, vp]
                L.ptc_session_lru_curves_workspace_bytes.restype = sz
                L.ptc_session_lru_curves_workspace_bytes.argtypes = [u64, u32, u32]
                L.ptc_session_lru_curves.restype = st
                L.ptc_session_lru_curves.argtypes = [vp, u64, u64, vp, vp, u32, u32, u32, ctypes.POINTER(CostModel),
                                                     vp, u32, vp, vp, vp, sz, vp]
                L.ptc_belady_curves_workspace_bytes.restype = sz
                L.ptc_belady_curves_workspace_bytes.argtypes = [u64, u32, u32]
                L.ptc_belady_curves.restype = st
                L.ptc_belady_curves.argtypes = [vp, u64, vp, u32, u32, ctypes.POINTER(CostModel), vp, u32, vp, vp, vp,
                                                vp, sz, vp]
                L.ptc_assign_ids_ex_workspace_bytes.restype = sz
                L.ptc_assign_ids_ex_workspace_bytes.argtypes = [u64, u32, ctypes.c_int]
                L.ptc_assign_ids_ex.restype = st
                L.ptc_assign_ids_ex.argtypes = [vp, u64, vp, vp, u32, vp, ctypes.POINTER(u64), ctypes.c_int, vp, sz, vp]
                L.ptc_assign_ids_prior_workspace_bytes.restype = sz
                L.ptc_assign_ids_prior_workspace_bytes.argtypes = [u64, u32]
                L.ptc_assign_ids_prior.restype = st
                L.ptc_assign_ids_prior.argtypes = [vp, u64, vp, vp, u32, vp, ctypes.POINTER(u64), vp, sz, vp]
                L.ptc_session_prior_workspace_bytes.restype = sz
                L.ptc_session_prior_workspace_bytes.argtypes = [u32]
                L.ptc_session_prior.restype = st
                L.ptc_session_prior.argtypes = [vp, u32, u32, vp, vp, sz, vp]
                L.ptc_stack_distance_variant_workspace_bytes.restype = sz
                L.ptc_stack_distance_variant_workspace_bytes.argtypes = [u64, u32, ctypes.c_int, ctypes.c_int]
                L.ptc_stack_distance_variant.restype = st
                L.ptc_stack_distance_variant.argtypes = [vp, u64, vp, u32, ctypes.c_int, ctypes.c_int, vp, vp, sz, vp]
                L.ptc_stack_distance_variant_ex.restype = st
                L.ptc_stack_distance_variant_ex.argtypes = [vp, u64, vp, u32, ctypes.c_int, ctypes.c_int, vp,
                                                            ctypes.c_int, vp, sz, vp]
                L.ptc_trace_stats_workspace_bytes.restype = sz
                L.ptc_trace_stats_workspace_bytes.argtypes = [u64, u64, u32, u32]
                L.ptc_trace_stats.restype = st
                L.ptc_trace_stats.argtypes = [vp, vp, vp, vp, u64, u64, vp, vp, vp, u32, u32, vp, u32, vp, vp, vp,
                                              sz, vp]
                L.ptc_release_host_staging.restype = None
                L.ptc_release_host_staging.argtypes = []
                L.ptc_test_wait_polls.restype = None
                L.ptc_test_wait_polls.argtypes = [u32]
                L.ptc_timer_enable.restype = None
                L.ptc_timer_enable.argtypes = [ctypes.c_int]
                L.ptc_timer_reset.restype = None
                L.ptc_timer_reset.argtypes = []
                L.ptc_timer_read.restype = u32
                L.ptc_timer_read.argtypes = [vp, u32]
                L.ptc_launch_count.restype = u64
                L.ptc_launch_count.argtypes = []
                del i64
                _lib = L
    return _lib


def version() -> str:
    return lib().ptc_version().decode()


def _check(call: str, rc: int):
    if rc != 0:
        raise PtcError(call, rc)


def _dev(t: torch.Tensor) -> torch.device:
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    return t.device


def _stream(device) -> int:
    return torch.cuda.current_stream(device).cuda_stream


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _workspace(nbytes: int, device, ws: torch.Tensor | None = None) -> torch.Tensor:
    nbytes = max(int(nbytes), 256)
    if ws is not None and ws.numel() >= nbytes and ws.device == device:
        return ws
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def u32(t: torch.Tensor) -> np.ndarray:
    """A host numpy uint32 view of an int32 tensor's bits."""
    return t.detach().cpu().numpy().view(np.uint32)


def u64(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy().view(np.uint64)


def to_device_u32(a, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).to(device)


def to_device_u64(a, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint64).view(np.int64)).to(device)


# ---------------------------------------------------------------- the five calls
def ptc_hash_blocks(tokens: torch.Tensor, req_tok_off: torch.Tensor, req_ts_us: torch.Tensor | None,
                    block_size: int, seed: int, keys_cap: int | None = None, ws: torch.Tensor | None = None):
    """Chained block keys.  Returns (keys int64[N, 2], req_blk_off int64[R+1], N)."""
    dev = _dev(req_tok_off)
    n_req = req_tok_off.numel() - 1
    n_tok = tokens.numel()
    cap = n_tok // block_size if keys_cap is None else int(keys_cap)
    keys = torch.empty((max(cap, 1), 2), dtype=torch.int64, device=dev)
    blk_off = torch.empty(n_req + 1, dtype=torch.int64, device=dev)
    need = lib().ptc_hash_blocks_workspace_bytes(n_req, n_tok, block_size)
    w = _workspace(need, dev, ws)
    n = ctypes.c_uint64(0)
    rc = lib().ptc_hash_blocks(_ptr(tokens), n_tok, _ptr(req_tok_off), _ptr(req_ts_us), n_req, block_size,
                               int(seed) & (2**64 - 1), _ptr(keys), cap, _ptr(blk_off), ctypes.byref(n),
                               _ptr(w), w.numel(), _stream(dev))
    _check("ptc_hash_blocks", rc)
    return keys[: n.value], blk_off, int(n.value)


def ptc_assign_ids(keys: torch.Tensor, ws: torch.Tensor | None = None):
    """Dense ids in first-occurrence order.  Returns (ids int32[N], D)."""
    dev = _dev(keys)
    n = keys.shape[0]
    ids = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    d = ctypes.c_uint64(0)
    w = _workspace(lib().ptc_assign_ids_workspace_bytes(n), dev, ws)
    rc = lib().ptc_assign_ids(_ptr(keys), n, _ptr(ids), ctypes.byref(d), _ptr(w), w.numel(), _stream(dev))
    _check("ptc_assign_ids", rc)
    return ids[:n], int(d.value)


def ptc_belady_curves(prev: torch.Tensor, req_blk_off: torch.Tensor, block_size: int, caps,
                      kind: int = PTC_COST_MEASURED, f_lin: int = F_LIN, f_attn: int = F_ATTN,
                      ws: torch.Tensor | None = None) -> dict:
    """Belady's MIN curves from the reuse indices.  Returns hits, saved
    (Python ints, exact) and raw_hits (without the prefix rule) per capacity."""
    dev = _dev(req_blk_off)
    n = prev.numel()
    R = req_blk_off.numel() - 1
    caps = np.ascontiguousarray(caps, dtype=np.uint64)
    G = caps.shape[0]
    w = _workspace(lib().ptc_belady_curves_workspace_bytes(n, R, G), dev, ws)
    hits = np.zeros(G, dtype=np.uint64)
    raw = np.zeros(G, dtype=np.uint64)
    saved = np.zeros(2 * G, dtype=np.uint64)
    cm = CostModel(int(f_lin), int(f_attn), int(kind))
    rc = lib().ptc_belady_curves(_ptr(prev), n, _ptr(req_blk_off), R, block_size, ctypes.byref(cm), caps.ctypes.data,
                                 G, hits.ctypes.data, saved.ctypes.data, raw.ctypes.data, _ptr(w), w.numel(),
                                 _stream(dev))
    _check("ptc_belady_curves", rc)
    return {"hits": [int(h) for h in hits], "raw_hits": [int(x) for x in raw],
            "saved": [int(saved[2 * g + 1]) << 64 | int(saved[2 * g]) for g in range(G)]}


def ptc_session_lru_curves(ids: torch.Tensor, n_distinct: int, req_blk_off: torch.Tensor, req_session: torch.Tensor,
                           n_session: int, block_size: int, caps, kind: int = PTC_COST_MEASURED, f_lin: int = F_LIN,
                           f_attn: int = F_ATTN, ws: torch.Tensor | None = None) -> dict:
    """Session-level LRU curves.  Returns hits and saved (Python ints, exact)."""
    dev = _dev(req_blk_off)
    n = ids.numel()
    R = req_blk_off.numel() - 1
    caps = np.ascontiguousarray(caps, dtype=np.uint64)
    G = caps.shape[0]
    w = _workspace(lib().ptc_session_lru_curves_workspace_bytes(n_distinct, n_session, G), dev, ws)
    hits = np.zeros(G, dtype=np.uint64)
    saved = np.zeros(2 * G, dtype=np.uint64)
    cm = CostModel(int(f_lin), int(f_attn), int(kind))
    rc = lib().ptc_session_lru_curves(_ptr(ids), n, int(n_distinct), _ptr(req_blk_off), _ptr(req_session), R,
                                      int(n_session), block_size, ctypes.byref(cm), caps.ctypes.data, G,
                                      hits.ctypes.data, saved.ctypes.data, _ptr(w), w.numel(), _stream(dev))
    _check("ptc_session_lru_curves", rc)
    return {"hits": [int(h) for h in hits],
            "saved": [int(saved[2 * g + 1]) << 64 | int(saved[2 * g]) for g in range(G)]}


def ptc_assign_ids_prior(keys: torch.Tensor, req_blk_off: torch.Tensor, req_prior: torch.Tensor,
                         ws: torch.Tensor | None = None):
    """Dense ids with a prior-request hint (req_prior[r] < r or PTC_NONE, int32
    CUDA tensor).  Returns (ids int32[N], D); the same ids as ptc_assign_ids."""
    dev = _dev(keys)
    n = keys.shape[0]
    R = req_prior.numel()
    ids = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    d = ctypes.c_uint64(0)
    w = _workspace(lib().ptc_assign_ids_prior_workspace_bytes(n, R), dev, ws)
    rc = lib().ptc_assign_ids_prior(_ptr(keys), n, _ptr(req_blk_off), _ptr(req_prior), R, _ptr(ids), ctypes.byref(d),
                                    _ptr(w), w.numel(), _stream(dev))
    _check("ptc_assign_ids_prior", rc)
    return ids[:n], int(d.value)


def ptc_assign_ids_ex(keys: torch.Tensor, method: int, req_blk_off: torch.Tensor | None = None,
                      req_prior: torch.Tensor | None = None, ws: torch.Tensor | None = None):
    """Dense ids by the named dedup method (PTC_IDS_AUTO / PTC_IDS_TABLE /
    PTC_IDS_PARTITIONED), with the prior-request hint when req_blk_off and
    req_prior are given.  Returns (ids int32[N], D)."""
    dev = _dev(keys)
    n = keys.shape[0]
    R = req_prior.numel() if req_prior is not None else 0
    ids = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    d = ctypes.c_uint64(0)
    w = _workspace(lib().ptc_assign_ids_ex_workspace_bytes(n, R, method), dev, ws)
    rc = lib().ptc_assign_ids_ex(_ptr(keys), n, _ptr(req_blk_off) if R else None, _ptr(req_prior) if R else None, R,
                                 _ptr(ids), ctypes.byref(d), method, _ptr(w), w.numel(), _stream(dev))
    _check("ptc_assign_ids_ex", rc)
    return ids[:n], int(d.value)


def ptc_session_prior(req_session: torch.Tensor, n_session: int, ws: torch.Tensor | None = None) -> torch.Tensor:
    """The previous request of each request's session (PTC_NONE for a
    session's first): int32 CUDA tensor of req_session's length."""
    dev = _dev(req_session)
    R = req_session.numel()
    out = torch.empty(max(R, 1), dtype=torch.int32, device=dev)
    w = _workspace(lib().ptc_session_prior_workspace_bytes(R), dev, ws)
    rc = lib().ptc_session_prior(_ptr(req_session), R, int(n_session), _ptr(out), _ptr(w), w.numel(), _stream(dev))
    _check("ptc_session_prior", rc)
    return out[:R]


def ptc_verify_ids(tokens, req_tok_off, req_blk_off, block_size: int, ids: torch.Tensor, n_distinct: int,
                   ws: torch.Tensor | None = None) -> None:
    """Exact check of ids against tokens; raises PtcError(PTC_ERR_HASH_COLLISION)."""
    dev = _dev(ids)
    n = ids.numel()
    w = _workspace(lib().ptc_verify_ids_workspace_bytes(n, n_distinct), dev, ws)
    rc = lib().ptc_verify_ids(_ptr(tokens), tokens.numel(), _ptr(req_tok_off), _ptr(req_blk_off), req_tok_off.numel() - 1,
                              block_size, _ptr(ids), n, n_distinct, _ptr(w), w.numel(), _stream(dev))
    _check("ptc_verify_ids", rc)


def ptc_reuse_indices(ids: torch.Tensor, n_distinct: int, ws: torch.Tensor | None = None, method: int | None = None):
    """Previous / next use of every access.  Returns (prev int32[N], next int32[N]).
    ``method`` (PTC_REUSE_AUTO / PTC_REUSE_SORT / PTC_REUSE_RUNS) goes through
    ptc_reuse_indices_ex; None calls ptc_reuse_indices."""
    dev = _dev(ids)
    n = ids.numel()
    prev = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    nxt = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    if method is None:
        w = _workspace(lib().ptc_reuse_indices_workspace_bytes(n, n_distinct), dev, ws)
        rc = lib().ptc_reuse_indices(_ptr(ids), n, n_distinct, _ptr(prev), _ptr(nxt), _ptr(w), w.numel(),
                                     _stream(dev))
        _check("ptc_reuse_indices", rc)
    else:
        w = _workspace(lib().ptc_reuse_indices_ex_workspace_bytes(n, n_distinct, method), dev, ws)
        rc = lib().ptc_reuse_indices_ex(_ptr(ids), n, n_distinct, _ptr(prev), _ptr(nxt), method, _ptr(w), w.numel(),
                                        _stream(dev))
        _check("ptc_reuse_indices_ex", rc)
    return prev[:n], nxt[:n]


def ptc_stack_distance(prev: torch.Tensor, ws: torch.Tensor | None = None, method: int | None = None) -> torch.Tensor:
    """LRU stack distance of every access (1-based; PTC_NONE for a first access).
    ``method`` (PTC_SD_AUTO / PTC_SD_POINTS / PTC_SD_RUNS) picks the wavelet
    matrix through ptc_stack_distance_ex; None calls ptc_stack_distance."""
    dev = _dev(prev)
    n = prev.numel()
    dist = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    if method is None:
        w = _workspace(lib().ptc_stack_distance_workspace_bytes(n), dev, ws)
        rc = lib().ptc_stack_distance(_ptr(prev), n, _ptr(dist), _ptr(w), w.numel(), _stream(dev))
        _check("ptc_stack_distance", rc)
    else:
        w = _workspace(lib().ptc_stack_distance_ex_workspace_bytes(n, method), dev, ws)
        rc = lib().ptc_stack_distance_ex(_ptr(prev), n, _ptr(dist), method, _ptr(w), w.numel(), _stream(dev))
        _check("ptc_stack_distance_ex", rc)
    return dist[:n]


def ptc_stack_distance_variant(prev: torch.Tensor, req_blk_off: torch.Tensor, touch_order: int, residency: int,
                               ws: torch.Tensor | None = None, method: int | None = None) -> torch.Tensor:
    """Stack distances under a touch order (PTC_TOUCH_*) and a residency rule
    (PTC_RESIDENCY_*), in root-first access order, ready for ptc_curves.
    ``method`` (PTC_SD_AUTO / PTC_SD_POINTS / PTC_SD_RUNS) picks the route for
    per-request residency through ptc_stack_distance_variant_ex."""
    dev = _dev(req_blk_off)
    n = prev.numel()
    n_req = req_blk_off.numel() - 1
    dist = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    w = _workspace(lib().ptc_stack_distance_variant_workspace_bytes(n, n_req, touch_order, residency), dev, ws)
    if method is None:
        rc = lib().ptc_stack_distance_variant(_ptr(prev), n, _ptr(req_blk_off), n_req, touch_order, residency,
                                              _ptr(dist), _ptr(w), w.numel(), _stream(dev))
    else:
        rc = lib().ptc_stack_distance_variant_ex(_ptr(prev), n, _ptr(req_blk_off), n_req, touch_order, residency,
                                                 _ptr(dist), method, _ptr(w), w.numel(), _stream(dev))
    _check("ptc_stack_distance_variant", rc)
    return dist[:n]


def ptc_curves(dist: torch.Tensor, req_blk_off: torch.Tensor, block_size: int, caps, kind: int = PTC_COST_MEASURED,
               f_lin: int = F_LIN, f_attn: int = F_ATTN, ws: torch.Tensor | None = None) -> dict:
    """Hit and compute-saved curves over the capacity grid ``caps`` (blocks).

    Returns {"hits": [int], "saved": [int], "total_cost": int} with exact
    integers (the 128-bit sums joined)."""
    dev = _dev(req_blk_off)
    n = dist.numel()
    caps = np.ascontiguousarray(caps, dtype=np.uint64)
    G = caps.shape[0]
    hits = np.zeros(G, dtype=np.uint64)
    saved = np.zeros(2 * G, dtype=np.uint64)
    total = U128()
    cm = CostModel(int(f_lin), int(f_attn), int(kind))
    w = _workspace(lib().ptc_curves_workspace_bytes(n, req_blk_off.numel() - 1, G), dev, ws)
    rc = lib().ptc_curves(_ptr(dist), n, _ptr(req_blk_off), req_blk_off.numel() - 1, block_size, ctypes.byref(cm),
                          caps.ctypes.data, G, hits.ctypes.data, saved.ctypes.data, ctypes.byref(total),
                          _ptr(w), w.numel(), _stream(dev))
    _check("ptc_curves", rc)
    return {"hits": [int(h) for h in hits],
            "saved": [int(saved[2 * g + 1]) << 64 | int(saved[2 * g]) for g in range(G)],
            "total_cost": int(total.hi) << 64 | int(total.lo)}


# ptc_trace_summary, field by field (all uint64, in declaration order):
# category-major histograms have 3 rows (0 shared across sessions, 1 session
# history, 2 single-turn), log2 histograms 65 bins (the bit length of the
# value), freq 256 exact bins with the blocks used 256 times or more in bin 0.
STAT_FIELDS = (("blocks", (3,)), ("accesses", (3,)), ("freq", (3, 256)), ("freq_log2", (3, 65)),
               ("reuse_us", (3, 65)), ("lifetime_us", (3, 65)), ("reuse_by_freq", (65, 65)),
               ("lifetime_by_freq", (65, 65)), ("dist_log2", (65,)), ("sess_requests", (65,)),
               ("sess_duration_us", (65,)))
STAT_SCALARS = ("n_access", "n_distinct", "n_reuse", "n_sessions", "n_multi_sessions")
STAT_WORDS = sum(int(np.prod(sh)) for _, sh in STAT_FIELDS) + len(STAT_SCALARS)


class TraceStatsPlan:
    """ptc_trace_stats with its arguments marshalled once: ``run()`` is one C
    call that rereads the given device arrays, ``result()`` converts the
    summary.  ``req_session`` is an int32 tensor of session labels below
    ``n_session``; ``caps`` needs ``dist``."""

    def __init__(self, ids: torch.Tensor, prev: torch.Tensor, nxt: torch.Tensor, n_distinct: int,
                 req_blk_off: torch.Tensor, req_ts_us: torch.Tensor, req_session: torch.Tensor, n_session: int,
                 dist: torch.Tensor | None = None, caps=None, ws: torch.Tensor | None = None):
        dev = _dev(req_blk_off)
        n = ids.numel()
        n_req = req_blk_off.numel() - 1
        self.caps = np.ascontiguousarray([] if caps is None else caps, dtype=np.uint64)
        G = self.caps.shape[0]
        self.reach = np.zeros(max(G, 1), dtype=np.uint64)
        self.buf = np.zeros(STAT_WORDS, dtype=np.uint64)
        self.ws = _workspace(lib().ptc_trace_stats_workspace_bytes(n, n_distinct, n_req, n_session), dev, ws)
        self._keep = (ids, prev, nxt, req_blk_off, req_ts_us, req_session, dist)
        self._fn = lib().ptc_trace_stats
        self._args = (_ptr(ids), _ptr(prev), _ptr(nxt), _ptr(dist), n, n_distinct, _ptr(req_blk_off),
                      _ptr(req_ts_us), _ptr(req_session), n_req, n_session, self.caps.ctypes.data if G else None, G,
                      self.reach.ctypes.data if G else None, self.buf.ctypes.data, _ptr(self.ws), self.ws.numel(),
                      _stream(dev))

    def run(self) -> "TraceStatsPlan":
        rc = self._fn(*self._args)
        if rc != 0:
            raise PtcError("ptc_trace_stats", rc)
        return self

    def result(self) -> dict:
        out, at = {}, 0
        for name, shape in STAT_FIELDS:
            size = int(np.prod(shape))
            out[name] = self.buf[at: at + size].reshape(shape).copy()
            at += size
        out.update({k: int(v) for k, v in zip(STAT_SCALARS, self.buf[at:])})
        if self.caps.shape[0]:
            out["reach"] = self.reach[: self.caps.shape[0]].copy()
        return out


def ptc_trace_stats(ids: torch.Tensor, prev: torch.Tensor, nxt: torch.Tensor, n_distinct: int,
                    req_blk_off: torch.Tensor, req_ts_us: torch.Tensor, req_session: torch.Tensor, n_session: int,
                    dist: torch.Tensor | None = None, caps=None, ws: torch.Tensor | None = None) -> dict:
    """Trace statistics (block categories, frequency, lifetime, reuse-interval
    and session histograms; reuses reachable within each of ``caps``).
    Returns numpy uint64 arrays named as in STAT_FIELDS, the STAT_SCALARS as
    ints, and ``reach`` when ``caps`` is given (it needs ``dist``)."""
    return TraceStatsPlan(ids, prev, nxt, n_distinct, req_blk_off, req_ts_us, req_session, n_session, dist, caps,
                          ws).run().result()


def workspace_bytes(n_req: int, n_tok: int, block_size: int, n: int | None = None, n_cap: int = MAX_CAPACITIES) -> int:
    """Largest workspace any of the five calls needs for a trace of this size
    (N defaults to its upper bound n_tok // block_size)."""
    L = lib()
    n = n_tok // block_size if n is None else n
    return max(L.ptc_hash_blocks_workspace_bytes(n_req, n_tok, block_size), L.ptc_assign_ids_workspace_bytes(n),
               L.ptc_reuse_indices_workspace_bytes(n, n), L.ptc_stack_distance_workspace_bytes(n),
               L.ptc_curves_workspace_bytes(n, n_req, n_cap), L.ptc_verify_ids_workspace_bytes(n, n))


def pipeline(tokens, req_tok_off, req_ts_us, block_size: int, caps_for, kind: int = PTC_COST_MEASURED,
             seed: int = 0, f_lin: int = F_LIN, f_attn: int = F_ATTN, ws: torch.Tensor | None = None,
             keep: bool = True) -> dict:
    """All five calls on one trace resident on the GPU.  ``caps_for`` is the
    capacity grid, or a function of D (distinct blocks) returning it.  One
    workspace (``ws``, grown if too small) serves every call."""
    dev = _dev(req_tok_off)
    if ws is None:
        ws = _workspace(workspace_bytes(req_tok_off.numel() - 1, tokens.numel(), block_size), dev)
    keys, blk_off, n = ptc_hash_blocks(tokens, req_tok_off, req_ts_us, block_size, seed, ws=ws)
    ids, d = ptc_assign_ids(keys, ws=ws)
    prev, nxt = ptc_reuse_indices(ids, d, ws=ws)
    dist = ptc_stack_distance(prev, ws=ws)
    caps = caps_for(d) if callable(caps_for) else caps_for
    cur = ptc_curves(dist, blk_off, block_size, caps, kind, f_lin, f_attn, ws=ws)
    out = dict(n_access=n, n_distinct=d, caps=np.asarray(caps, dtype=np.uint64), **cur)
    if keep:
        out.update(keys=keys, req_blk_off=blk_off, ids=ids, prev=prev, next=nxt, dist=dist)
    return out


class PipelinePlan:
    """ptc_pipeline with its arguments marshalled once, for running the same
    call again and again (a serving loop, a benchmark): ``run()`` is one C
    call.  The device tensors given here are read at every run, so a new
    trace of the same shape is run by refilling them in place.  The stream is
    the current stream of the tensors' device when the plan is made.
    ``outputs`` may map any of keys / req_blk_off / ids / prev / next / dist to
    preallocated CUDA tensors that receive those arrays.  After ``run()``,
    ``hits`` (uint64, one per capacity) and ``saved`` (uint64 pairs lo, hi)
    hold the curves, and ``result()`` converts them as ptc_pipeline returns
    them."""

    def __init__(self, tokens, req_tok_off, req_ts_us, block_size: int, caps, kind: int = PTC_COST_MEASURED,
                 seed: int = 0, f_lin: int = F_LIN, f_attn: int = F_ATTN, ws: torch.Tensor | None = None,
                 outputs: dict | None = None, req_session: torch.Tensor | None = None, n_session: int = 0):
        dev = _dev(req_tok_off)
        n_req = req_tok_off.numel() - 1
        n_tok = tokens.numel()
        self.caps = np.ascontiguousarray(caps, dtype=np.uint64)
        G = self.caps.shape[0]
        self.ws = _workspace(lib().ptc_pipeline_workspace_bytes(n_req, n_tok, block_size, G), dev, ws)
        o = outputs or {}
        self.hits = np.zeros(G, dtype=np.uint64)
        self.saved = np.zeros(2 * G, dtype=np.uint64)
        self.total = U128()
        self.n, self.d = ctypes.c_uint64(0), ctypes.c_uint64(0)
        self.cm = CostModel(int(f_lin), int(f_attn), int(kind))
        self._keep = (tokens, req_tok_off, req_ts_us, req_session, o)  # the pointers below stay valid
        self._fn = lib().ptc_pipeline
        self._args = (_ptr(tokens), n_tok, _ptr(req_tok_off), _ptr(req_ts_us), _ptr(req_session),
                      int(n_session) if req_session is not None else 0, n_req, block_size,
                      int(seed) & (2**64 - 1), ctypes.byref(self.cm), self.caps.ctypes.data, G, _ptr(o.get("keys")),
                      _ptr(o.get("req_blk_off")), _ptr(o.get("ids")), _ptr(o.get("prev")), _ptr(o.get("next")),
                      _ptr(o.get("dist")), ctypes.byref(self.n), ctypes.byref(self.d), self.hits.ctypes.data,
                      self.saved.ctypes.data, ctypes.byref(self.total), _ptr(self.ws), self.ws.numel(), _stream(dev))

    def run(self) -> "PipelinePlan":
        rc = self._fn(*self._args)
        if rc != 0:
            raise PtcError("ptc_pipeline", rc)
        return self

    def result(self) -> dict:
        G = self.hits.shape[0]
        return {"n_access": int(self.n.value), "n_distinct": int(self.d.value), "hits": [int(h) for h in self.hits],
                "saved": [int(self.saved[2 * g + 1]) << 64 | int(self.saved[2 * g]) for g in range(G)],
                "total_cost": int(self.total.hi) << 64 | int(self.total.lo)}


class HostPipelinePlan:
    """ptc_pipeline_host with its arguments marshalled once: the trace is in
    host memory (numpy arrays or CPU tensors; page-locked memory copies at
    full speed) and every ``run()`` copies it to the device and runs the whole
    path in one C call on the current stream of ``device``.  The workspace
    (device memory, which also holds the copied trace) is made once.  After
    ``run()`` the fields are those of PipelinePlan."""

    def __init__(self, tokens, req_tok_off, req_ts_us, block_size: int, caps, kind: int = PTC_COST_MEASURED,
                 seed: int = 0, f_lin: int = F_LIN, f_attn: int = F_ATTN, device="cuda",
                 ws: torch.Tensor | None = None, req_session=None, n_session: int = 0):
        dev = torch.device(device)
        if dev.index is None:
            dev = torch.device("cuda", torch.cuda.current_device())

        def host_ptr(a, dt):
            if a is None:
                return None, None
            if isinstance(a, torch.Tensor):
                if a.is_cuda:
                    raise ValueError("HostPipelinePlan takes host buffers")
                return a, a.data_ptr()
            a = np.ascontiguousarray(a, dtype=dt)
            return a, a.ctypes.data

        tok, tp = host_ptr(tokens, np.uint32)
        off, op = host_ptr(req_tok_off, np.uint64)
        ts, sp = host_ptr(req_ts_us, np.int64)
        ses, sep = host_ptr(req_session, np.uint32)
        n_req = (off.numel() if isinstance(off, torch.Tensor) else off.shape[0]) - 1
        n_tok = tok.numel() if isinstance(tok, torch.Tensor) else tok.shape[0]
        self.caps = np.ascontiguousarray(caps, dtype=np.uint64)
        G = self.caps.shape[0]
        self.ws = _workspace(lib().ptc_pipeline_host_workspace_bytes(n_req, n_tok, block_size, G), dev, ws)
        self.hits = np.zeros(G, dtype=np.uint64)
        self.saved = np.zeros(2 * G, dtype=np.uint64)
        self.total = U128()
        self.n, self.d = ctypes.c_uint64(0), ctypes.c_uint64(0)
        self.cm = CostModel(int(f_lin), int(f_attn), int(kind))
        self._keep = (tok, off, ts, ses)
        self._fn = lib().ptc_pipeline_host
        self._args = (tp, n_tok, op, sp, sep, int(n_session) if ses is not None else 0, n_req, block_size, int(seed) & (2**64 - 1), ctypes.byref(self.cm),
                      self.caps.ctypes.data, G, ctypes.byref(self.n), ctypes.byref(self.d), self.hits.ctypes.data,
                      self.saved.ctypes.data, ctypes.byref(self.total), _ptr(self.ws), self.ws.numel(), _stream(dev))

    def run(self) -> "HostPipelinePlan":
        rc = self._fn(*self._args)
        if rc != 0:
            raise PtcError("ptc_pipeline_host", rc)
        return self

    result = PipelinePlan.result


def ptc_pipeline(tokens, req_tok_off, req_ts_us, block_size: int, caps, kind: int = PTC_COST_MEASURED, seed: int = 0,
                 f_lin: int = F_LIN, f_attn: int = F_ATTN, ws: torch.Tensor | None = None, outputs: dict | None = None,
                 req_session: torch.Tensor | None = None, n_session: int = 0):
    """All five stages in one C call (trace already on the GPU).  ``outputs``
    may map any of keys / req_blk_off / ids / prev / next / dist to
    preallocated CUDA tensors that receive those arrays.  Returns the curves
    with N and D."""
    return PipelinePlan(tokens, req_tok_off, req_ts_us, block_size, caps, kind, seed, f_lin, f_attn, ws,
                        outputs, req_session, n_session).run().result()
