"""Host-side helpers of the bench, on the CPU.  The NUMA placement of the
page-locked token buffer of the end-to-end leg: its pages are asked for on
the GPU's NUMA node before they are touched; where the system names no node
(no GPU here, or a device sysfs does not describe), nothing is asked and the
buffer is placed as before.  And the algorithmic bytes the bench credits to
the partitioned dedup's kernels."""
import mmap
import os
import platform
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _untouched(nbytes=1 << 22):
    m = mmap.mmap(-1, nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
    return m, np.frombuffer(m, dtype=np.uint32)


@pytest.mark.skipif(platform.machine() not in ("x86_64", "aarch64") or not os.path.isdir("/sys/devices/system/node/node0"),
                    reason="needs Linux on x86_64 or aarch64 with NUMA node 0")
def test_prefer_node_zero_succeeds_and_pages_stay_usable():
    m, a = _untouched()
    assert bench.prefer_node(a.ctypes.data, len(m), 0)
    b = np.frombuffer(m, dtype=np.uint32)
    b[:] = np.arange(b.size, dtype=np.uint32)  # first touch under the policy
    assert int(b[-1]) == b.size - 1


def test_prefer_node_refuses_what_it_cannot_ask():
    m, a = _untouched()
    assert not bench.prefer_node(a.ctypes.data, len(m), None)
    assert not bench.prefer_node(a.ctypes.data, len(m), 4096)  # beyond the 1,024-node mask


def test_gpu_numa_node_without_a_gpu_is_none():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present: the node comes from its sysfs entry")
    assert bench.gpu_numa_node(0) is None


def test_partitioned_dedup_model_bytes():
    """The bench's algorithmic bytes for the partitioned dedup's kernels: per
    settled access U, 16 bytes for each pass that reads the records or the
    settled keys and 16 more for each that writes records, plus the bitmaps;
    nothing when U is not known."""
    T, N, L, D, U = 10_000, 1_000, 10, 400, 600
    want = {"k_pd_flags": N / 4, "k_pd_count": 16 * U + N / 8, "k_pd_scatter1": 32 * U + N / 8,
            "k_pd_count2": 16 * U, "k_pd_scatter2": 32 * U, "k_pd_dedup": 16 * U}
    for name, b in want.items():
        assert bench.kernel_model_bytes(name, T, N, L, D, U) == b
        assert bench.kernel_model_bytes(name, T, N, L, D) == 0.0
    assert bench.kernel_model_bytes("k_hash16", T, N, L, D, U) == 4 * T + 16 * N
    assert set(want) <= set(bench.PD_KERNELS)
