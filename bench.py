#!/usr/bin/env python3
"""Benchmark: request trace -> all-capacity LRU hit and compute-saved curves.

One step is the whole path — block hashing, dense ids, reuse indices, stack
distances, curves — in one ptc_pipeline call over one synthetic trace
resident in HBM.  The headline workload is the largest one that fits one GPU:
the mixed 24-hour trace (~10B tokens, ~624M block accesses, 16-token blocks,
128 log-spaced capacities from 0.1% to 100% of the distinct blocks,
measured-shape cost model).  The metric is trace tokens per second; the JSON
line also carries block accesses per second, the fraction of the HBM
roofline for the stage-byte model and for the path's own bytes, the dominant
kernel's roofline, the end-to-end rate through the host-buffer C call, and the
conversational chat trace (~154M tokens) as an extra key.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload 0-3] [--requests R]

Timing: W untimed warm-up steps, then K steps, each bracketed by CUDA events
on the launching stream, with a 256 MiB write between steps to flush L2
(outside the events); barrier + synchronize on both sides; max over ranks.
Per-kernel durations (for the roofline of the dominant kernel) come from a
second pass of K steps with events around every launch.
With N > 1 (torchrun) every rank runs an independent replica (the path has
no cross-GPU exchange): value = tokens of all replicas / slowest rank's time.

The CPU oracle (the plain restatement used as the parity reference) runs on
a bounded prefix of the same workload on the host cores, and the GPU path
runs on that prefix too: their curves must be equal (cpu_baseline).
--impl reference times that oracle alone, per step, on the prefix; rank 0
alone runs it.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "trace tokens/s to all-capacity LRU hit+compute-saved curves; % of HBM roofline"
WORKLOAD = 3   # the mixed 24-hour trace
CHAT = 1       # the conversational chat trace, reported as an extra key
BLOCK = 16
NOMINAL_HBM_GBS = 7900.0

# Per-launch DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) from
# the last ncu capture of each kernel, keyed by (kernel, workload), with the
# sha256 prefix of the source file it was taken on (a changed source reads as
# "no counters", null) and how the capture was scaled to a full launch.
NCU_TRAFFIC: dict[tuple[str, int], tuple[float, str, str]] = {
    ("k_hash16", 1): (6.3766e+08, "d33ef0cf44921375", "ncu dram__bytes metrics, first 6,000 requests, x 153.81 / 55.67"),
    ("k_hash16", 3): (4.9715e+10, "d33ef0cf44921375", "ncu dram__bytes metrics, first 60,000 requests: reads x tokens "
                      "(9984.4M / 943.9M), key writes x blocks (623.75M / 58.97M)"),
}


VARIANTS = (("leaf_first", 1, 0), ("request_residency", 0, 1), ("leaf_first_request_residency", 1, 1))


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", type=int, choices=[0, 1, 2, 3], default=WORKLOAD,
                    help="0 tiny, 1 chat, 2 agentic, 3 mixed 24 h (the headline)")
    ap.add_argument("--cpu-sample", type=float, default=None,
                    help="fraction of the workload's requests (a prefix in time) the CPU oracle runs on "
                         "(default: all of workloads 0-1, 5%% of 2-3)")
    ap.add_argument("--ref-sample", type=float, default=None,
                    help="fraction of requests per --impl reference step (default as --cpu-sample)")
    ap.add_argument("--json-out", default=None)
    ap.add_argument("--requests", type=int, default=0,
                    help="run only the first N requests of the workload (small cases for profiling)")
    ap.add_argument("--profile-one-step", action="store_true",
                    help="set up, run one warm-up step, then exactly one step between cudaProfilerStart and "
                         "cudaProfilerStop (for ncu --profile-from-start off), and exit")
    return ap.parse_args()


# ---------------------------------------------------------------- helpers
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x, world, device=None):
    """The largest x over the ranks of the default process group: the slowest
    replica's time.  x itself on one rank (no process group)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_step, steps, world, total_ms):
    """Units per second of the whole job: every replica processes the same
    units each step (weak scaling), and the job lasts as long as its slowest
    replica (total_ms, already the max over ranks)."""
    return world * units_per_step * steps / (total_ms * 1e-3)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def value_bits(n):  # values of the wavelet matrix lie in [0, n]
    L = 1
    while L < 33 and (1 << L) <= n:
        L += 1
    return L


def stage_model_bytes(T, N):
    """Algorithmic bytes of each stage (the stage-byte model)."""
    L = value_bits(N)
    return {
        "hash": 4 * T + 16 * N,
        "ids": 20 * N,
        "reuse": 12 * N,
        "wavelet_build": 8.125 * L * N,
        "queries": (8 + L / 8) * N,
        "curves": 4 * N,
    }, L


def sort_passes(D):
    b = 1
    while b < 32 and (1 << b) < D:
        b += 1
    return (b + 7) // 8


def kernel_model_bytes(name, T, N, L, D, U=None):
    """Algorithmic bytes one launch of `name` moves under the stage-byte model
    (0: the kernel only touches scratch the model does not count).  `U`: the
    accesses the partitioned dedup settles (those the prior-request hint does
    not match), for its kernels; None leaves them at 0."""
    per_level = ((L - 1) * 8.125 + 4.125) / L * N  # the last level writes no partition
    pd = {} if U is None else {
        "k_pd_flags": N / 4,               # the settled-access bitmap and its copy out
        "k_pd_count": 16 * U + N / 8,      # settled keys (whole 32-byte sectors) and the bitmap in
        "k_pd_scatter1": 32 * U + N / 8,   # settled keys in, bucket records out
        "k_pd_count2": 16 * U,             # records in
        "k_pd_scatter2": 32 * U,           # records in, partition records out
        "k_pd_dedup": 16 * U,              # records in
    }
    return {
        "k_hash_local": 4 * T + 16 * N,   # token stream in, block keys out
        "k_hash16": 4 * T + 16 * N,       # the same, B = 16 path
        "k_hash_tile": 4 * T + 16 * N,    # the same, other multiples of 16
        "k_ids_insert": 16 * N,           # keys in
        "k_ids_insert_prior": 16 * N,     # keys in (the same stage, prior-request hint)
        "k_ids_gather": 4 * N,            # ids out
        "k_sort_scatter": 12 * N / sort_passes(D),  # ids in, prev / next out, spread over the passes
        "k_ir_count": 4 * N,              # ids in (sort over id-runs)
        "k_ir_fill": 8 * N,               # prev / next out (sort over id-runs)
        "k_wm_level": per_level,          # values in, partition + bit plane out
        "k_wm_heads": (8 + L / 8) * N,    # prev in, one read of the bit planes, distances out
        "k_runs_mark": 4 * N,             # prev in (matrix over runs)
        "k_runs_expand": 4 * N,           # distances out (matrix over runs)
        "k_curves": 4 * N,                # distances in
        **pd,
    }.get(name, 0.0)


KERNEL_SOURCE = {
    "k_block_offsets": "ptc_hash.cu", "k_pow_tables": "ptc_hash.cu", "k_hash_local": "ptc_hash.cu",
    "k_hash16": "ptc_hash.cu", "k_hash_tile": "ptc_hash.cu", "k_fill_many": "ptc_abi.cu",
    "k_hash_chain": "ptc_hash.cu", "k_ids_insert": "ptc_ids.cu",
    "k_ids_gather": "ptc_ids.cu", "k_ids_insert_prior": "ptc_ids.cu", "k_ids_follow": "ptc_ids.cu",
    "k_tile_req": "ptc_ids.cu", "k_ids_lam": "ptc_ids.cu", "k_session_prior": "ptc_ids.cu", "k_sort_count": "ptc_sort.cu", "k_sort_rowscan": "ptc_sort.cu",
    "k_sort_scatter": "ptc_sort.cu", "k_sort_links": "ptc_sort.cu", "k_ir_count": "ptc_reuse.cu",
    "k_ir_mark": "ptc_reuse.cu", "k_bm_count": "ptc_reuse.cu", "k_bm_words": "ptc_reuse.cu",
    "k_ir_inc1": "ptc_reuse.cu", "k_ir_inc2": "ptc_reuse.cu", "k_ir_fill": "ptc_reuse.cu", "k_wm_count0": "ptc_wavelet.cu",
    "k_wm_level": "ptc_wavelet.cu", "k_wm_dir": "ptc_wavelet.cu", "k_wm_heads": "ptc_wavelet.cu",
    "k_wm_propagate": "ptc_wavelet.cu", "k_runs_mark": "ptc_runs.cu", "k_runs_count": "ptc_runs.cu", "k_runs_init": "ptc_runs.cu",
    "k_runs_level": "ptc_runs.cu", "k_runs_build_cluster": "ptc_runs.cu", "k_runs_query": "ptc_runs.cu", "k_runs_expand": "ptc_runs.cu", "k_heads": "ptc_curves.cu", "k_curves_agg": "ptc_curves.cu",
    "k_curves": "ptc_curves.cu", "k_finalize": "ptc_curves.cu", "k_curves_fast": "ptc_curves.cu",
    "k_curves_runs": "ptc_curves.cu", "k_fill": "ptc_abi.cu", "k_copy_words": "ptc_abi.cu",
    "k_copy_err": "ptc_abi.cu", "k_carry_err": "ptc_abi.cu", "k_hash_carry": "ptc_hash.cu",
    "k_rank_count": "ptc_abi.cu", "k_rank_words": "ptc_abi.cu", "k_pd_flags": "ptc_ids.cu",
    "k_pd_count": "ptc_ids.cu", "k_pd_rows1": "ptc_ids.cu", "k_pd_scatter1": "ptc_ids.cu",
    "k_pd_count2": "ptc_ids.cu", "k_pd_rows2": "ptc_ids.cu", "k_pd_scatter2": "ptc_ids.cu", "k_pd_dedup": "ptc_ids.cu",
}


def source_sha(kernel):
    f = KERNEL_SOURCE.get(kernel)
    if f is None:
        return None
    with open(os.path.join(ROOT, "paper_2609_28870_gb300", "csrc", f), "rb") as fh:
        return hashlib.sha256(fh.read()).hexdigest()[:16]


class Clocks:
    """nvidia-smi sampled every 200 ms while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "", 1).isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "", 1).isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4) if r[5 + k].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------- our arm
WORKLOAD_NAMES = {
    0: "tiny conversational trace (workload 0, seed 0): 444 sessions, 16-point capacity grid",
    1: "conversational chat trace (workload 1, seed 1): 5,600 sessions, 60% single-turn, LN(300)/LN(600) turns, "
       "50 Zipf system prompts, B=16, 64-point capacity grid, measured-shape cost",
    2: "agentic coding trace (workload 2, seed 2): 560 sessions, Zipf(1.2) turns <= 400, 131,072-token cap, B=16, "
       "64-point capacity grid, measured-shape cost",
    3: "mixed 24 h trace (workload 3, seed 3): 50/50 token mix of the chat and agentic generators, diurnal arrivals "
       "(3x peak/trough), ~10B tokens, ~624M block accesses, fully resident, B=16, 128-point capacity grid from "
       "0.1% to 100% of distinct blocks, measured-shape cost",
}
GOLDEN = os.path.join(ROOT, "tests", "golden", "big_configs.json")


_HOST_BUFFERS = []  # registered host buffers: kept alive, unregistered at exit
HOST_PLACEMENT = {}  # where the token buffer's pages were asked to live (reported with e2e)


def gpu_numa_node(dev):
    """The host NUMA node of the GPU's PCI device (sysfs numa_node), or None
    where the system does not say."""
    try:
        import torch
        p = torch.cuda.get_device_properties(dev)
        path = f"/sys/bus/pci/devices/{p.pci_domain_id:04x}:{p.pci_bus_id:02x}:{p.pci_device_id:02x}.0/numa_node"
        with open(path) as fh:
            node = int(fh.read().strip())
        return node if node >= 0 else None
    except Exception:
        return None


def prefer_node(addr, nbytes, node):
    """Asks the kernel to place the pages of [addr, addr + nbytes), not yet
    touched, on NUMA node `node` (mbind with MPOL_PREFERRED: other nodes
    still serve it when that one is full).  True if the call succeeded."""
    import ctypes
    import platform
    nr = {"aarch64": 235, "x86_64": 237}.get(platform.machine())
    if nr is None or node is None or node >= 1024:
        return False
    try:
        libc = ctypes.CDLL(None, use_errno=True)
        libc.syscall.restype = ctypes.c_long
        mask = (ctypes.c_ulong * 16)()
        mask[node // 64] |= 1 << (node % 64)
        mpol_preferred = 1
        rc = libc.syscall(ctypes.c_long(nr), ctypes.c_void_p(addr), ctypes.c_ulong(nbytes),
                          ctypes.c_int(mpol_preferred), mask, ctypes.c_ulong(16 * 64 + 1), ctypes.c_uint(0))
        return rc == 0
    except Exception:
        return False


def registered_host_u32(n, dev=None):
    """n uint32 in page-locked host memory: an anonymous mapping asked for huge
    pages (and, where the system names the GPU's NUMA node, for pages on that
    node: the copy engine reads a far node's memory through the link between
    the CPUs), then registered with CUDA (cudaHostRegister).  End-to-end steps
    over this buffer measured 226-250 ms on some boxes and 305-569 ms on
    others before the node was asked for; a buffer from torch's pinned-memory
    allocator copied at 84-211 GB/s on its first passes."""
    import atexit
    import mmap

    import numpy as np
    import torch
    nbytes = max(4 * int(n), 4096)
    m = mmap.mmap(-1, nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
    a = np.frombuffer(m, dtype=np.uint32, count=int(n))
    node = gpu_numa_node(dev) if dev is not None else None
    HOST_PLACEMENT.update({"gpu_numa_node": node, "placed": prefer_node(a.ctypes.data, nbytes, node)})
    if hasattr(mmap, "MADV_HUGEPAGE"):
        m.madvise(mmap.MADV_HUGEPAGE)
    rt = torch.cuda.cudart()
    if int(rt.cudaHostRegister(a.ctypes.data, nbytes, 0)) != 0:
        raise RuntimeError("cudaHostRegister failed for the token buffer")
    _HOST_BUFFERS.append((m, a))
    if len(_HOST_BUFFERS) == 1:
        atexit.register(lambda: [rt.cudaHostUnregister(b.ctypes.data) for _, b in _HOST_BUFFERS])
    return a


def load_trace(workload, requests, dev):
    """The workload generated into page-locked host memory (the end-to-end leg
    copies from it) and copied once to the device."""
    import numpy as np
    import torch
    import tracegen
    if requests:
        tr = tracegen.make(workload, max_requests=requests)
        tok_host = torch.from_numpy(tr.tokens.view(np.int32)).pin_memory()
    else:
        _, T, _ = tracegen.sizes(workload)
        buf = registered_host_u32(T, dev)
        tr = tracegen.make(workload, token_buffer=buf)
        tok_host = torch.from_numpy(buf.view(np.int32))
    off_host = torch.from_numpy(tr.req_tok_off.view(np.int64)).pin_memory()
    ts_host = torch.from_numpy(tr.req_ts_us).pin_memory()
    ses_host = torch.from_numpy(np.ascontiguousarray(tr.req_session, dtype=np.uint32).view(np.int32)).pin_memory()
    dev_t = (tok_host.to(dev, non_blocking=True), off_host.to(dev, non_blocking=True),
             ts_host.to(dev, non_blocking=True), ses_host.to(dev, non_blocking=True))
    torch.cuda.synchronize(dev)
    return tr, (tok_host, off_host, ts_host, ses_host), dev_t


def grid_for(ptc, tracegen, workload, dev_t, n_req, T):
    """D is a property of the trace, taken once before timing; the grid spans
    the workload's range over it."""
    import torch
    tok, off, ts, _ = dev_t
    ws = torch.empty(ptc.workspace_bytes(n_req, T, BLOCK, n_cap=1), dtype=torch.uint8, device=tok.device)
    D = ptc.pipeline(tok, off, ts, BLOCK, lambda d: [1], ws=ws, keep=False)["n_distinct"]
    del ws
    return D, tracegen.workload_grid(workload, D)


class Timer:
    """CUDA events on the launch stream around each step, an L2 flush (a
    256 MiB write) between steps outside the events, and a check that every
    step returns the warm-up's curves."""

    def __init__(self, dev, stream):
        import torch
        self.flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        self.stream = stream

    def run(self, k_steps, body, plan=None, ref=None):
        import numpy as np
        import torch
        ms = []
        for k in range(k_steps):
            self.flush.fill_(k & 0xFF)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(self.stream)
            body()
            e1.record(self.stream)
            e1.synchronize()
            ms.append(e0.elapsed_time(e1))
            if plan is not None:
                assert np.array_equal(plan.hits, ref[0]) and np.array_equal(plan.saved, ref[1])
        return ms


def kernel_table(ktimes, steps, T, N, D, Lbits, U=None):
    kernels = []
    for name, launches_k, tot_ms in ktimes:
        per = tot_ms / max(launches_k, 1)
        mb = kernel_model_bytes(name, T, N, Lbits, D, U)
        kernels.append({"name": name, "launches_per_step": launches_k / steps, "ms_per_step": tot_ms / steps,
                        "avg_launch_ms": per, "model_bytes_per_launch": mb,
                        "achieved_gbs": (mb / (per * 1e-3) / 1e9) if per > 0 else 0.0})
    kernels.sort(key=lambda x: -x["ms_per_step"])
    return kernels


def roofline_of(kernels, peak, peak_kind, workload):
    """The dominant kernel's algorithmic bytes over its average launch time."""
    if not kernels:
        return None
    dom = kernels[0]
    tr_entry = NCU_TRAFFIC.get((dom["name"], workload))
    traffic = tr_entry[0] if tr_entry and tr_entry[1] == source_sha(dom["name"]) else None
    return {"kernel": dom["name"], "bound": "hbm", "achieved": round(dom["achieved_gbs"], 1), "peak": peak,
            "unit": "GB/s", "frac": round(dom["achieved_gbs"] / peak, 4), "traffic": traffic,
            "traffic_source": tr_entry[2] if traffic is not None else None,
            "peak_source": f"{peak_kind} hbm_gbs"}


def hint_matched(ptc, torch, ids, blk_off, ses):
    """Accesses the prior-request hint matches (their block equals the block
    at the same depth of the previous request of their session): the id
    table's insert probes the others.  Counted from the step's ids."""
    R = ses.numel()
    order = torch.sort(ses.to(torch.int64), stable=True).indices
    ss = ses.to(torch.int64)[order]
    prior_sorted = torch.full((R,), -1, dtype=torch.int64, device=ids.device)
    prior_sorted[1:] = torch.where(ss[1:] == ss[:-1], order[:-1], torch.full_like(order[:-1], -1))
    prior = torch.empty_like(prior_sorted)
    prior[order] = prior_sorted
    n_r = blk_off[1:] - blk_off[:-1]
    matched = 0
    step = 1 << 16  # requests per slice: bounded temporaries
    for r0 in range(0, R, step):
        r1 = min(R, r0 + step)
        cnt = n_r[r0:r1]
        req = torch.repeat_interleave(torch.arange(r0, r1, device=ids.device), cnt)
        k = torch.arange(int(cnt.sum()), device=ids.device) - torch.repeat_interleave(
            torch.cumsum(cnt, 0) - cnt, cnt)
        p = prior[req]
        ok = (p >= 0) & (k < n_r[p.clamp(min=0)])
        i = blk_off[req] + k
        j = blk_off[p.clamp(min=0)] + k
        eq = ok & (ids[i] == ids[j.clamp(max=ids.numel() - 1)])
        matched += int(eq.sum())
    return matched


PD_KERNELS = ("k_pd_flags", "k_pd_count", "k_pd_rows1", "k_pd_scatter1", "k_pd_count2", "k_pd_rows2",
              "k_pd_scatter2", "k_pd_dedup")


def id_stage(ptc, torch, L, kernels, n_access, matched, peak, dev):
    """The partitioned dedup's kernels against the measured copy bandwidth
    (they stream their records), and, for comparison, the time a hash table
    of DRAM size would need at best: the accesses it settles at the rate
    this GPU completes random 16-byte read-modify-writes on such a table,
    measured in this run (ptc_probe_random_rmw)."""
    pd = [k for k in kernels if k["name"] in PD_KERNELS]
    if not pd:
        return None
    settled = n_access - matched
    ms = sum(k["avg_launch_ms"] for k in pd)
    mb = sum(k["model_bytes_per_launch"] for k in pd)
    slots = 1
    while slots < n_access // 4 * 3 + 64:  # the table method's first size for a DRAM-sized table
        slots *= 2
    table = torch.empty(slots * 2, dtype=torch.int64, device=dev)
    sink = torch.zeros(1, dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    best = None
    for rep in range(3):
        table.fill_(-1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        rc = L.ptc_probe_random_rmw(table.data_ptr(), slots, settled, 0x5EED + rep, sink.data_ptr(), stream.cuda_stream)
        e1.record(stream)
        e1.synchronize()
        if rc != 0:
            raise RuntimeError(f"ptc_probe_random_rmw failed ({rc})")
        t = e0.elapsed_time(e1)
        best = t if best is None else min(best, t)
    del table, sink
    achieved = mb / (ms * 1e-3) / 1e9
    return {"method": "partitioned dedup (65,536 partitions by 16 key bits, shared-memory tables)",
            "settled": settled, "matched_by_hint": matched, "ms": round(ms, 4),
            "model_bytes": int(mb), "achieved_gbs": round(achieved, 1), "peak": peak,
            "frac": round(achieved / peak, 4),
            "kernels_ms": {k["name"]: round(k["avg_launch_ms"], 4) for k in pd},
            "table_bound_ms": round(best, 4),
            "table_bound_how": "ptc_probe_random_rmw in this run: one random 16-byte slot load plus a 128-bit CAS "
                               f"claim per settled access, on an all-ones table of {slots * 16 / 1e9:.2f} GB; best "
                               "of 3 (a lower bound for the hash-table method's insert)"}


def hbm_fractions(T, N, ms, peak):
    stages, Lbits = stage_model_bytes(T, N)
    model_total = sum(stages.values())
    own = 4 * T + 60 * N
    sec = ms * 1e-3
    return {"stage_model_bytes": model_total, "L": Lbits,
            "frac_of_measured": round(model_total / sec / 1e9 / peak, 4),
            "frac_of_nominal_7900": round(model_total / sec / 1e9 / NOMINAL_HBM_GBS, 4),
            "path_bytes_4T_60N": own, "path_frac_of_measured": round(own / sec / 1e9 / peak, 4),
            "stages_bytes": stages}, Lbits


def golden_parity(workload, N, D, hits, saved, caps):
    """The full-size headline curves against the oracle's stored results
    (tests/golden/big_configs.json, written by a script that runs the oracle
    alone), where an entry for this workload exists."""
    key = {3: "mixed_B16", 2: "agentic_B16"}.get(workload)
    if key is None or not os.path.exists(GOLDEN):
        return None
    with open(GOLDEN) as f:
        g = json.load(f).get(key)
    if g is None:
        return None
    same = (g["N"] == N and g["D"] == D and g["caps"] == [int(c) for c in caps]
            and g["hits"] == [int(h) for h in hits] and g["saved"] == [str(int(s)) for s in saved])
    return {"golden": f"tests/golden/big_configs.json[{key}]", "equal": bool(same)}


def run_ours(args, ws_world, rank, local):
    import numpy as np
    import torch

    import paper_2609_28870_gb300 as ptc
    import tracegen

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws_world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        if ws_world > 1:
            import torch.distributed as dist
            dist.barrier()

    def slowest(x):
        return max_over_ranks(x, ws_world, dev)

    L = ptc.lib()
    W = args.workload
    stream = torch.cuda.current_stream(dev)
    timer = Timer(dev, stream)
    peak, peak_kind = measured_peaks()

    # ================================================= the headline workload
    tr, host_t, dev_t = load_trace(W, args.requests, dev)
    T, R = tr.n_tok, tr.n_req
    D, caps = grid_for(ptc, tracegen, W, dev_t, R, T)
    G = len(caps)
    tok, off, ts, ses = dev_t
    ws = torch.empty(L.ptc_pipeline_workspace_bytes(R, T, BLOCK, G), dtype=torch.uint8, device=dev)
    # the call a serving loop makes: arguments marshalled once, one C call per step
    plan = ptc.PipelinePlan(tok, off, ts, BLOCK, caps, kind=ptc.PTC_COST_MEASURED, seed=0, ws=ws,
                            req_session=ses, n_session=tr.n_sessions)
    for _ in range(max(args.warmup, 0)):
        plan.run()
    N = plan.n.value
    ref = (plan.hits.copy(), plan.saved.copy())
    if args.profile_one_step:
        torch.cuda.synchronize(dev)
        launches0 = L.ptc_launch_count()
        torch.cuda.profiler.start()
        plan.run()
        torch.cuda.synchronize(dev)
        torch.cuda.profiler.stop()
        assert np.array_equal(plan.hits, ref[0]) and np.array_equal(plan.saved, ref[1])
        if rank == 0:
            print(json.dumps({"profiled_step": WORKLOAD_NAMES[W], "tokens": T, "accesses": N,
                              "launches": L.ptc_launch_count() - launches0}), flush=True)
        return

    # ---- timed region (inputs resident in HBM)
    clocks = Clocks(local)
    barrier()
    torch.cuda.synchronize(dev)
    clocks.start()
    launches0 = L.ptc_launch_count()
    step_ms = timer.run(args.steps, plan.run, plan, ref)
    torch.cuda.synchronize(dev)
    launches = L.ptc_launch_count() - launches0
    barrier()
    clk = clocks.stop()
    total_ms = slowest(sum(step_ms))
    ms_per_step = total_ms / args.steps

    # ---- per-kernel durations: the same K steps again with CUDA events
    # around every launch on the launch stream (the events slow a step, so
    # this pass is separate from the timed one)
    L.ptc_timer_reset()
    L.ptc_timer_enable(1)
    inst_ms = timer.run(args.steps, plan.run, plan, ref)
    L.ptc_timer_enable(0)
    ktimes = read_timer(ptc)
    hbm, Lbits = hbm_fractions(T, N, ms_per_step, peak)
    # the accesses the prior-request hint matches (one more step with the
    # ids kept): the partitioned dedup settles the others
    matched = None
    if any(name in PD_KERNELS for name, _, _ in ktimes):
        ids_t = torch.empty(N, dtype=torch.int32, device=dev)
        boff_t = torch.empty(R + 1, dtype=torch.int64, device=dev)
        ptc.PipelinePlan(tok, off, ts, BLOCK, caps, kind=ptc.PTC_COST_MEASURED, seed=0, ws=ws,
                         outputs={"ids": ids_t, "req_blk_off": boff_t}, req_session=ses,
                         n_session=tr.n_sessions).run()
        matched = hint_matched(ptc, torch, ids_t, boff_t, ses)
        del ids_t, boff_t
    kernels = kernel_table(ktimes, args.steps, T, N, D, Lbits, None if matched is None else N - matched)
    roof = roofline_of(kernels, peak, peak_kind, W)
    gold = golden_parity(W, N, D, plan.hits, plan.result()["saved"], caps) if not args.requests else None
    ids_summary = id_stage(ptc, torch, L, kernels, N, matched, peak, dev) if matched is not None else None
    del plan, ws, tok, off, ts, ses, dev_t
    torch.cuda.empty_cache()

    # ---- end to end through the C ABI with HOST buffers: each step copies
    # the trace from page-locked host memory to the device inside the call,
    # runs the path and returns the curves to host memory
    hplan = ptc.HostPipelinePlan(*host_t[:3], BLOCK, caps, kind=ptc.PTC_COST_MEASURED, seed=0, device=dev,
                                 req_session=host_t[3], n_session=tr.n_sessions)
    for _ in range(max(args.warmup, 3)):  # the first copies out of a new page-locked buffer run slow
        hplan.run()
    assert np.array_equal(hplan.hits, ref[0]) and np.array_equal(hplan.saved, ref[1])
    e2e_total = slowest(sum(timer.run(args.steps, hplan.run, hplan, ref)))
    h2d = 4 * T + 8 * (R + 1) + 8 * R + 4 * R
    d2h = 8 * G + 16 * G + 16 + 8 + 8  # hits, saved (u128), total cost, N, D
    del hplan
    torch.cuda.empty_cache()

    value = whole_job_rate(T, args.steps, ws_world, total_ms)
    acc_s = whole_job_rate(N, args.steps, ws_world, total_ms)
    e2e_value = whole_job_rate(T, args.steps, ws_world, e2e_total)
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws_world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u32/u64 integer", "data": "synthetic",
        "config": {"workload": WORKLOAD_NAMES[W], "tokens": T, "requests": R, "accesses": N, "distinct_blocks": D,
                   "block_size": BLOCK, "capacities": G,
                   "l2": "inputs larger than L2; also flushed between timed steps (256 MiB write, outside the events)",
                   "parallelism": "replicas" if ws_world > 1 else "single GPU",
                   "prefix_requests": args.requests or None},
        "accesses_per_s": round(acc_s, 1),
        "hbm_roofline": hbm,
        "roofline": roof,
        "kernels": [{k: (round(v, 5) if isinstance(v, float) else v) for k, v in x.items()} for x in kernels],
        "kernel_timing": {"how": "separate pass of the same K steps with CUDA events around every launch",
                          "ms_per_step": round(sum(inst_ms) / len(inst_ms), 4)},
        "e2e": {"value": round(e2e_value, 1), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_total / args.steps, 4),
                "call": "ptc_pipeline_host: trace in page-locked host memory, copied inside the call; curves "
                        "returned to host memory",
                "host_pages": dict(HOST_PLACEMENT) or None},
        "gpu_launches": launches,
        "clocks": clk,
        "parity_with_oracle_golden": gold,
        "id_stage": ids_summary,
    }

    # ---- the oracle on a bounded prefix of the same workload, and the GPU
    # on that same prefix: the curves must be equal
    if rank == 0 and ws_world == 1 and not args.no_cpu_baseline:
        frac = args.cpu_sample if args.cpu_sample is not None else (1.0 if W in (0, 1) else 0.05)
        cb, orc = cpu_baseline(tr, frac, W)
        cb["parity_with_gpu"] = gpu_matches_oracle(ptc, orc, dev)
        assert cb["parity_with_gpu"], "the GPU's curves differ from the oracle's on the sample"
        line["cpu_baseline"] = cb
    del tr, host_t
    torch.cuda.empty_cache()

    # ================================================= the chat trace (an extra key)
    if W != CHAT and not args.requests:
        line["chat"] = chat_extras(args, ptc, tracegen, dev, timer, slowest, peak, peak_kind, rank, ws_world)
    if rank == 0:
        s = json.dumps(line)
        print(s, flush=True)
        if args.json_out:
            with open(args.json_out, "w") as f:
                f.write(s + "\n")
    if ws_world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def gpu_matches_oracle(ptc, orc, dev):
    """Run the GPU path on the oracle's sample trace and compare N, D, the
    curves and the total cost with the oracle's."""
    import numpy as np
    import torch
    sub = orc["sub"]
    tok = torch.from_numpy(sub.tokens.view(np.int32)).to(dev)
    off = torch.from_numpy(sub.req_tok_off.view(np.int64)).to(dev)
    ts = torch.from_numpy(sub.req_ts_us).to(dev)
    ses = torch.from_numpy(np.ascontiguousarray(sub.req_session, dtype=np.uint32).view(np.int32)).to(dev)
    g = ptc.ptc_pipeline(tok, off, ts, BLOCK, orc["caps"], kind=ptc.PTC_COST_MEASURED, req_session=ses,
                         n_session=sub.n_sessions)
    return bool(g["n_access"] == orc["n"] and g["n_distinct"] == orc["D"] and g["hits"] == orc["hits"]
                and g["saved"] == orc["saved"] and g["total_cost"] == orc["total"])


def chat_extras(args, ptc, tracegen, dev, timer, slowest, peak, peak_kind, rank, ws_world):
    """The conversational chat trace (~154M tokens) through the same path,
    its oracle parity on the whole trace, and the trace statistics and
    semantics variants over its per-access arrays."""
    import numpy as np
    import torch
    L = ptc.lib()
    tr, host_t, dev_t = load_trace(CHAT, 0, dev)
    T, R = tr.n_tok, tr.n_req
    D, caps = grid_for(ptc, tracegen, CHAT, dev_t, R, T)
    G = len(caps)
    tok, off, ts, ses_d = dev_t
    ws = torch.empty(L.ptc_pipeline_workspace_bytes(R, T, BLOCK, G), dtype=torch.uint8, device=dev)
    plan = ptc.PipelinePlan(tok, off, ts, BLOCK, caps, kind=ptc.PTC_COST_MEASURED, seed=0, ws=ws,
                            req_session=ses_d, n_session=tr.n_sessions)
    for _ in range(max(args.warmup, 0)):
        plan.run()
    N = plan.n.value
    ref = (plan.hits.copy(), plan.saved.copy())
    ms = slowest(sum(timer.run(args.steps, plan.run, plan, ref))) / args.steps
    L.ptc_timer_reset()
    L.ptc_timer_enable(1)
    timer.run(args.steps, plan.run, plan, ref)
    L.ptc_timer_enable(0)
    hbm, Lbits = hbm_fractions(T, N, ms, peak)
    kernels = kernel_table(read_timer(ptc), args.steps, T, N, D, Lbits)
    out = {"workload": WORKLOAD_NAMES[CHAT], "tokens": T, "requests": R, "accesses": N, "distinct_blocks": D,
           "capacities": G, "ms_per_step": round(ms, 4), "tokens_per_s": round(ws_world * T / (ms * 1e-3), 1),
           "accesses_per_s": round(ws_world * N / (ms * 1e-3), 1), "hbm_roofline": hbm,
           "roofline": roofline_of(kernels, peak, peak_kind, CHAT),
           "kernels_top": [{"name": k["name"], "ms_per_step": round(k["ms_per_step"], 4)} for k in kernels[:8]]}
    # ---- trace statistics (Sec. 4.1-4.3, App. B) over the path's own
    # per-access arrays: one pipeline run that keeps them, then K timed calls
    outs = {k: torch.empty(max(N, 1), dtype=torch.int32, device=dev) for k in ("ids", "prev", "next", "dist")}
    outs["req_blk_off"] = torch.empty(R + 1, dtype=torch.int64, device=dev)
    ptc.PipelinePlan(tok, off, ts, BLOCK, caps, ws=ws, outputs=outs, req_session=ses_d,
                     n_session=tr.n_sessions).run()
    ses = torch.from_numpy(tr.req_session.astype(np.uint32).view(np.int32)).to(dev)
    splan = ptc.TraceStatsPlan(outs["ids"][:N], outs["prev"][:N], outs["next"][:N], D, outs["req_blk_off"], ts, ses,
                               tr.n_sessions, dist=outs["dist"][:N], caps=caps)
    stats = splan.run().result()
    assert stats["n_reuse"] == N - D and int(stats["blocks"].sum()) == D and int(stats["accesses"].sum()) == N
    L.ptc_timer_reset()
    L.ptc_timer_enable(1)
    splan.run()
    L.ptc_timer_enable(0)
    st_kernels = {name: round(tot, 4) for name, _, tot in read_timer(ptc)}
    st_ms = slowest(sum(timer.run(args.steps, splan.run))) / args.steps
    out["trace_stats"] = {
        "call": "ptc_trace_stats on the step's ids, prev, next and stack distances, 64-point reach grid",
        "ms": round(st_ms, 4), "accesses_per_s": round(ws_world * N / (st_ms * 1e-3), 1),
        "roofline": {"bound": "hbm", "bytes_model": "16 N: ids, prev, next, dist read once",
                     "achieved": round(16 * N / (st_ms * 1e-3) / 1e9, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(16 * N / (st_ms * 1e-3) / 1e9 / peak, 4), "traffic": None},
        "kernels_ms": st_kernels,
        "categories": {"blocks": stats["blocks"].tolist(), "accesses": stats["accesses"].tolist(),
                       "one_hit_blocks": [int(stats["freq"][c, 1]) for c in range(3)]},
    }
    # ---- semantics variants (Sec. 3.1): stack distances under leaf-first
    # touch order and whole-request residency from the step's prev, then the
    # curves on them
    variants, vdists = {}, {}
    prev_t, rbo = outs["prev"][:N], outs["req_blk_off"]
    mid = [0, G // 2, G - 1]
    for vname, order, res in VARIANTS:
        vws = torch.empty(L.ptc_stack_distance_variant_workspace_bytes(N, R, order, res), dtype=torch.uint8,
                          device=dev)
        vdist = torch.empty(max(N, 1), dtype=torch.int32, device=dev)
        vargs = (prev_t.data_ptr(), N, rbo.data_ptr(), R, order, res, vdist.data_ptr(), vws.data_ptr(),
                 vws.numel(), timer.stream.cuda_stream)

        def vrun(vargs=vargs):
            rc = L.ptc_stack_distance_variant(*vargs)
            assert rc == 0, rc

        vrun()
        v_ms = slowest(sum(timer.run(args.steps, vrun))) / args.steps
        cur = ptc.ptc_curves(vdist[:N], rbo, BLOCK, caps)
        variants[vname] = {"touch_order": "leaf-first" if order else "root-first",
                           "residency": "per request" if res else "per block", "ms": round(v_ms, 4),
                           "achieved_gbs_8n": round(8 * N / (v_ms * 1e-3) / 1e9, 1),
                           "hit_ratio_at": {str(int(caps[g])): round(cur["hits"][g] / N, 5) for g in mid}}
        vdists[vname] = (order, res, vdist[:N])
        del vws
    out["variants"] = {"call": "ptc_stack_distance_variant on the step's prev (distances in depth order for "
                               "ptc_curves)", "bytes_model": "8 N: prev read, dist written",
                       "hot_path_hit_ratio_at": {str(int(caps[g])): round(int(plan.hits[g]) / N, 5) for g in mid},
                       **variants}
    # ---- Belady's offline optimum (Sec. 3.2) from the step's prev, every grid capacity
    bws = torch.empty(L.ptc_belady_curves_workspace_bytes(N, R, G), dtype=torch.uint8, device=dev)
    bel = ptc.ptc_belady_curves(prev_t, rbo, BLOCK, caps, ws=bws)
    L.ptc_timer_reset()
    L.ptc_timer_enable(1)
    ptc.ptc_belady_curves(prev_t, rbo, BLOCK, caps, ws=bws)
    L.ptc_timer_enable(0)
    bel_kernels = {name: round(tot, 4) for name, _, tot in read_timer(ptc)}
    bel_ms = slowest(sum(timer.run(args.steps, lambda: ptc.ptc_belady_curves(prev_t, rbo, BLOCK, caps, ws=bws)))) \
        / args.steps
    del bws
    out["belady"] = {"call": "ptc_belady_curves on the step's prev: MIN curves at every grid capacity, one warp per "
                             "capacity over runs of re-reads", "ms": round(bel_ms, 3), "kernels_ms": bel_kernels,
                     "hit_ratio_at": {str(int(caps[g])): round(bel["hits"][g] / N, 5) for g in mid},
                     "lru_hit_ratio_at": {str(int(caps[g])): round(int(plan.hits[g]) / N, 5) for g in mid}}
    # ---- session-level eviction (Sec. 5.3) on the step's ids, every grid capacity
    ses_t = ses
    sws = torch.empty(L.ptc_session_lru_curves_workspace_bytes(D, tr.n_sessions, G), dtype=torch.uint8, device=dev)
    ids_t = outs["ids"][:N]
    sesc = ptc.ptc_session_lru_curves(ids_t, D, rbo, ses_t, tr.n_sessions, BLOCK, caps, ws=sws)
    ses_ms = slowest(sum(timer.run(args.steps, lambda: ptc.ptc_session_lru_curves(
        ids_t, D, rbo, ses_t, tr.n_sessions, BLOCK, caps, ws=sws)))) / args.steps
    del sws
    out["session_eviction"] = {
        "call": "ptc_session_lru_curves on the step's ids: session-level LRU at every grid capacity, one warp per "
                "capacity", "ms": round(ses_ms, 3),
        "hit_ratio_at": {str(int(caps[g])): round(sesc["hits"][g] / N, 5) for g in mid},
        "block_level_hit_ratio_at": {str(int(caps[g])): round(int(plan.hits[g]) / N, 5) for g in mid}}
    if rank == 0 and ws_world == 1 and not args.no_cpu_baseline:
        # the oracle on the whole chat trace: curves, statistics and variant distances must match
        cb, orc = cpu_baseline(tr, 1.0, CHAT, keep_sd=True)
        g_res = plan.result()
        same = (orc["n"] == N and orc["D"] == D and orc["hits"] == g_res["hits"] and orc["saved"] == g_res["saved"]
                and orc["total"] == g_res["total_cost"])
        assert same, "the chat trace's curves differ from the oracle's"
        cb["parity_with_gpu"] = same
        out["cpu_baseline"] = cb
        ost, odt = oracle_trace_stats(tr, orc)
        same_st = all(np.array_equal(np.asarray(ost[k]), np.asarray(stats[k])) for k in ost)
        assert same_st, "trace statistics differ from the oracle"
        out["trace_stats"]["cpu_baseline"] = {
            "value": round(orc["n"] / odt, 1), "unit": "accesses/s", "cores": 1, "kind": "oracle",
            "sample": f"orc_trace_stats on the oracle's own ids and distances of the whole trace "
                      f"({orc['n']} accesses); {odt:.2f} s", "parity_with_gpu": same_st}
        import oracle
        for vname, (order, res, vd) in vdists.items():
            t0 = time.perf_counter()
            want = oracle.sd_variant(orc["ids"], orc["D"], orc["off"], order, res)
            dt = time.perf_counter() - t0
            same_v = bool(np.array_equal(ptc.u32(vd), want))
            assert same_v, f"variant {vname} differs from the oracle"
            out["variants"][vname]["cpu_baseline"] = {
                "value": round(N / dt, 1), "unit": "accesses/s", "cores": 1, "kind": "oracle",
                "sample": f"orc_sd_variant (Fenwick) on the whole trace; {dt:.2f} s", "parity_with_gpu": same_v}
        threads = os.cpu_count() or 1
        t0 = time.perf_counter()
        bh, bs, braw = oracle.belady_curves(orc["ids"], orc["off"], BLOCK, caps, threads=threads)
        dt = time.perf_counter() - t0
        same_b = bh == bel["hits"] and bs == bel["saved"] and braw == bel["raw_hits"]
        assert same_b, "Belady curves differ from the oracle"
        t0 = time.perf_counter()
        sh_, ss_ = oracle.session_lru_curves(orc["ids"], orc["off"], tr.req_session.astype(np.uint32), tr.n_sessions,
                                             BLOCK, caps, threads=threads)
        dts = time.perf_counter() - t0
        same_s = sh_ == sesc["hits"] and ss_ == sesc["saved"]
        assert same_s, "session-level curves differ from the oracle"
        out["session_eviction"]["cpu_baseline"] = {
            "value": round(N / dts, 1), "unit": "accesses/s", "cores": threads, "kind": "oracle",
            "sample": f"orc_session_lru_curves (direct simulation per capacity) on the whole trace, all {G} "
                      f"capacities; {dts:.2f} s", "parity_with_gpu": same_s}
        out["belady"]["cpu_baseline"] = {
            "value": round(N / dt, 1), "unit": "accesses/s", "cores": threads, "kind": "oracle",
            "sample": f"orc_belady_curves (direct MIN per capacity) on the whole trace, all {G} capacities; "
                      f"{dt:.2f} s", "parity_with_gpu": same_b}
    return out


def read_timer(ptc):
    import ctypes

    class KT(ctypes.Structure):
        _fields_ = [("name", ctypes.c_char * 48), ("launches", ctypes.c_uint64), ("total_ms", ctypes.c_double)]

    L = ptc.lib()
    L.ptc_timer_read.restype = ctypes.c_uint32
    L.ptc_timer_read.argtypes = [ctypes.c_void_p, ctypes.c_uint32]
    n = L.ptc_timer_read(None, 0)
    buf = (KT * max(n, 1))()
    n = L.ptc_timer_read(ctypes.cast(buf, ctypes.c_void_p), n)
    return [(buf[i].name.decode(), int(buf[i].launches), float(buf[i].total_ms)) for i in range(n)]


# ---------------------------------------------------------------- CPU oracle
def oracle_on_sample(tr, fraction, threads, workload, keep=False):
    """The oracle as it stands on the first `fraction` of the requests:
    exact trie ids, prev / next, Fenwick stack distances, direct LRU
    simulation at every capacity of the workload's grid over the sample's D."""
    import oracle
    import tracegen
    n_req = max(1, int(tr.n_req * fraction))
    sub = tr.head(n_req)
    t0 = time.perf_counter()
    ids, D = oracle.block_ids(sub.tokens, sub.req_tok_off, BLOCK)
    off = oracle.block_offsets(sub.req_tok_off, BLOCK)
    prev, nxt = oracle.reuse(ids, D)
    sd = oracle.sd_fenwick(prev)
    caps = tracegen.workload_grid(workload, D)
    hits, saved, total = oracle.lru_curves(ids, off, BLOCK, caps, oracle.COST_MEASURED, threads=threads)
    dt = time.perf_counter() - t0
    res = dict(sub=sub, D=D, n=int(ids.size), n_req=n_req, caps=caps, hits=hits, saved=saved, total=total)
    if keep:
        res.update(ids=ids, off=off, sd=sd)
    return sub, dt, res


def cpu_baseline(tr, fraction, workload, keep_sd=False):
    threads = os.cpu_count() or 1
    sub, dt, res = oracle_on_sample(tr, fraction, threads, workload, keep=keep_sd)
    line = {"value": round(sub.n_tok / dt, 1), "unit": "tokens/s", "cores": threads, "kind": "oracle",
            "sample": f"first {sub.n_req} of {tr.n_req} requests ({sub.n_tok} tokens, {res['n']} accesses) of the "
                      f"same workload; exact trie ids, prev/next, Fenwick stack distances, direct LRU simulation "
                      f"at all {len(res['caps'])} capacities of the workload's grid over the sample's D on "
                      f"{threads} threads; {dt:.2f} s"}
    return line, res


def oracle_trace_stats(tr, kept):
    """The oracle's trace statistics on its own arrays of the sample, timed."""
    import oracle
    sub = kept["sub"]
    caps = kept["caps"] if kept["n_req"] == tr.n_req else None
    t0 = time.perf_counter()
    st = oracle.trace_stats(kept["ids"], kept["D"], kept["off"], sub.req_ts_us, sub.req_session, tr.n_sessions,
                            kept["sd"], caps)
    return st, time.perf_counter() - t0


def run_reference(args, ws_world, rank):
    if rank != 0:
        return
    import tracegen
    W = args.workload
    frac = args.ref_sample if args.ref_sample is not None else (1.0 if W in (0, 1) else 0.05)
    tr = tracegen.make(W, max_requests=max(1, int(tracegen.sizes(W)[0] * frac)))
    threads = os.cpu_count() or 1
    for _ in range(max(args.warmup, 0)):
        oracle_on_sample(tr, 1.0, threads, W)
    times = []
    sub = None
    for _ in range(args.steps):
        sub, dt, _ = oracle_on_sample(tr, 1.0, threads, W)
        times.append(dt)
    total = sum(times)
    value = sub.n_tok * args.steps / total
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws_world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(1e3 * total / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u32/u64/u128 integer", "data": "synthetic",
        "impl": "reference",
        "config": {"workload": WORKLOAD_NAMES[W], "sample_requests": sub.n_req, "sample_tokens": sub.n_tok},
        "cpu_baseline": {"value": round(value, 1), "unit": "tokens/s", "cores": threads, "kind": "oracle",
                         "sample": f"first {sub.n_req} requests ({sub.n_tok} tokens) of the workload per step: "
                                   f"exact trie ids, prev/next, Fenwick stack distances, direct LRU at every "
                                   f"capacity of the grid"},
        "e2e": {"value": round(value, 1), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    s = json.dumps(line)
    print(s, flush=True)
    if args.json_out:
        with open(args.json_out, "w") as f:
            f.write(s + "\n")


def main():
    args = parse_args()
    ws_world, rank, local = dist_env()
    if args.impl == "reference":
        run_reference(args, ws_world, rank)
    else:
        run_ours(args, ws_world, rank, local)


if __name__ == "__main__":
    main()
