"""The C-ABI library: it builds for sm_103a, loads, and exports every
function that include/ptc.h declares.  No GPU work is launched here."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libptc():
    from paper_2609_28870_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def declared_functions():
    src = open(os.path.join(ROOT, "include", "ptc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ptc_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_five_calls():
    names = declared_functions()
    for n in ("ptc_hash_blocks", "ptc_assign_ids", "ptc_reuse_indices", "ptc_stack_distance", "ptc_curves"):
        assert n in names and n + "_workspace_bytes" in names


def test_every_declared_symbol_is_exported(libptc):
    for name in declared_functions():
        assert hasattr(libptc, name), name


def test_strerror_and_version(libptc):
    libptc.ptc_strerror.restype = ctypes.c_char_p
    libptc.ptc_version.restype = ctypes.c_char_p
    assert libptc.ptc_strerror(0) == b"ok"
    assert b"timestamps" in libptc.ptc_strerror(2)
    assert b"sm_103a" in libptc.ptc_version()


def test_workspace_sizes_are_host_only_and_grow(libptc):
    f = libptc.ptc_stack_distance_workspace_bytes
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.c_uint64]
    assert 0 < f(1000) < f(10**6) < f(10**8)
    g = libptc.ptc_hash_blocks_workspace_bytes
    g.restype = ctypes.c_size_t
    g.argtypes = [ctypes.c_uint32, ctypes.c_uint64, ctypes.c_uint32]
    assert g(10, 10**6, 16) % 256 == 0


def test_host_argument_checks_need_no_gpu(libptc):
    """Bad arguments are rejected before any CUDA call."""
    import paper_2609_28870_gb300 as ptc
    L = ptc.lib()
    n = ctypes.c_uint64(0)
    # block size 0 and above the maximum
    for B in (0, ptc.MAX_BLOCK_SIZE + 1):
        rc = L.ptc_hash_blocks(None, 0, 8, None, 1, B, 0, None, 0, 8, ctypes.byref(n), None, 0, None)
        assert rc == 1
    # workspace missing
    rc = L.ptc_stack_distance(8, 10, 8, None, 0, None)
    assert rc == 4
    # too many accesses for 32-bit indices
    assert L.ptc_stack_distance(8, 2**32 - 1, 8, None, 0, None) == 3


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    import paper_2609_28870_gb300 as ptc
    monkeypatch.setattr(ptc, "_lib", None)
    monkeypatch.setattr(ptc._build, "LIB", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        ptc.lib()


def test_trace_summary_layout_matches_binding(tmp_path):
    """The binding reads ptc_trace_summary as a flat uint64 array: every
    field's offset and the struct's size, as a C compiler lays them out."""
    import subprocess
    import numpy as np
    import paper_2609_28870_gb300 as ptc
    fields = [n for n, _ in ptc.STAT_FIELDS] + list(ptc.STAT_SCALARS)
    src = tmp_path / "layout.c"
    src.write_text("#include <stdio.h>\n#include <stddef.h>\n#include \"ptc.h\"\nint main(void) {\n"
                   + "".join(f'  printf("%zu\\n", offsetof(ptc_trace_summary, {f}));\n' for f in fields)
                   + '  printf("%zu\\n", sizeof(ptc_trace_summary));\n  return 0;\n}\n')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    want, at = [], 0
    for _, shape in ptc.STAT_FIELDS:
        want.append(8 * at)
        at += int(np.prod(shape))
    for _ in ptc.STAT_SCALARS:
        want.append(8 * at)
        at += 1
    assert got == want + [8 * ptc.STAT_WORDS]


def test_trace_stats_host_checks_need_no_gpu(libptc):
    """ptc_trace_stats rejects bad arguments before any CUDA call."""
    import numpy as np
    import paper_2609_28870_gb300 as ptc
    L = ptc.lib()
    buf = np.zeros(ptc.STAT_WORDS, dtype=np.uint64)
    caps = np.array([4, 2], dtype=np.uint64)
    reach = np.zeros(2, dtype=np.uint64)
    fake = 256  # never dereferenced: the checks below fail first
    # no output
    assert L.ptc_trace_stats(fake, fake, fake, fake, 10, 5, fake, fake, fake, 2, 2, None, 0, None, None,
                             fake, 1 << 20, None) == 1
    # capacities not ascending
    assert L.ptc_trace_stats(fake, fake, fake, fake, 10, 5, fake, fake, fake, 2, 2, caps.ctypes.data, 2,
                             reach.ctypes.data, buf.ctypes.data, fake, 1 << 20, None) == 1
    # capacities without distances
    caps2 = np.array([2, 4], dtype=np.uint64)
    assert L.ptc_trace_stats(fake, fake, fake, None, 10, 5, fake, fake, fake, 2, 2, caps2.ctypes.data, 2,
                             reach.ctypes.data, buf.ctypes.data, fake, 1 << 20, None) == 1
    # more distinct blocks than accesses; N at the marker
    assert L.ptc_trace_stats(fake, fake, fake, None, 10, 11, fake, fake, fake, 2, 2, None, 0, None,
                             buf.ctypes.data, fake, 1 << 20, None) == 1
    assert L.ptc_trace_stats(fake, fake, fake, None, 0xFFFFFFFF, 5, fake, fake, fake, 2, 2, None, 0, None,
                             buf.ctypes.data, fake, 1 << 20, None) == 3
    # workspace too small
    assert L.ptc_trace_stats(fake, fake, fake, None, 10, 5, fake, fake, fake, 2, 2, None, 0, None,
                             buf.ctypes.data, fake, 16, None) == 4


def test_assign_ids_ex_checks_and_workspace(libptc):
    """An unknown dedup method is rejected before any CUDA call; the
    partitioned method's workspace holds its records and counters."""
    import paper_2609_28870_gb300 as ptc
    L = ptc.lib()
    d = ctypes.c_uint64(0)
    assert L.ptc_assign_ids_ex(None, 0, None, None, 0, None, ctypes.byref(d), 7, None, 0, None) == 1
    w = L.ptc_assign_ids_ex_workspace_bytes
    n = 100_000
    assert w(n, 0, ptc.PTC_IDS_PARTITIONED) > w(n, 0, ptc.PTC_IDS_TABLE)
    assert w(n, 0, ptc.PTC_IDS_PARTITIONED) >= 32 * n                       # records of both levels
    assert w(n, 0, ptc.PTC_IDS_AUTO) == w(n, 0, ptc.PTC_IDS_TABLE)        # small: the table
    big = 50_000_000
    assert w(big, 0, ptc.PTC_IDS_AUTO) == w(big, 0, ptc.PTC_IDS_PARTITIONED)  # beyond L2: partitions
    assert w(big, 0, ptc.PTC_IDS_AUTO) == L.ptc_assign_ids_workspace_bytes(big)


def test_probe_random_rmw_rejects_bad_tables(libptc):
    """Argument checks come before any CUDA call."""
    f = libptc.ptc_probe_random_rmw
    f.restype = ctypes.c_int
    f.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p]
    invalid = 1
    assert f(None, 1024, 10, 0, 256, None) == invalid            # no table
    assert f(4096, 1000, 10, 0, 256, None) == invalid            # slots not a power of two
    assert f(4104, 1024, 10, 0, 256, None) == invalid            # table not 16-byte aligned
    assert f(4096, 1024, 10, 0, 260, None) == invalid            # sink not 8-byte aligned
    assert f(4096, 1024, 0, 0, 256, None) == 0                   # no probes: nothing to do
