"""Host-side helpers of the bench's end-to-end leg, on the CPU: the NUMA
placement of the page-locked token buffer.  The buffer's pages are asked
for on the GPU's NUMA node before they are touched; where the system names no
node (no GPU here, or a device sysfs does not describe), nothing is asked
and the buffer is placed as before."""
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
