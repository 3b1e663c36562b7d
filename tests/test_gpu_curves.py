"""ptc_curves on hand-made distance arrays, against the definition written
out in Python: the running max of the distances over each request's blocks
(root-first), a hit at capacity C iff that max is <= C, and the 128-bit sum
of the depth-dependent cost over the hits.  Covers distances that fall
inside a request (where the running max binds) as well as the usual
non-decreasing case, for every cost kind."""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.gpu
NONE = 0xFFFFFFFF


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_28870_gb300 as ptc
    ptc.lib()


def _cost(k, B, kind, f_lin, f_attn):
    if kind == 0:
        return 1
    attn = f_attn * (B * B * k + B * (B + 1) // 2)
    return attn + (B * f_lin if kind == 1 else 0)


def _curves_by_definition(dist, blk_off, caps, B, kind, f_lin=oracle.F_LIN, f_attn=oracle.F_ATTN):
    hits = [0] * len(caps)
    saved = [0] * len(caps)
    total = 0
    for r in range(len(blk_off) - 1):
        e = 0
        for k, i in enumerate(range(int(blk_off[r]), int(blk_off[r + 1]))):
            e = max(e, int(dist[i]))
            c = _cost(k, B, kind, f_lin, f_attn)
            total += c
            for g, cap in enumerate(caps):
                if e != NONE and e <= cap:
                    hits[g] += 1
                    saved[g] += c
    return hits, saved, total


def _gpu_curves(dist, blk_off, caps, B, kind):
    import paper_2609_28870_gb300 as ptc
    d = ptc.to_device_u32(np.asarray(dist, dtype=np.uint32))
    off = ptc.to_device_u64(np.asarray(blk_off, dtype=np.uint64))
    return ptc.ptc_curves(d, off, B, caps, kind)


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("falls", [False, True])
def test_random_distances(seed, falls):
    rng = np.random.default_rng(seed * 2 + falls)
    R = int(rng.integers(1, 40))
    lens = rng.integers(0, 300, size=R)
    blk_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    n = int(blk_off[-1])
    dist = np.empty(n, dtype=np.uint64)
    for r in range(R):
        a, b = int(blk_off[r]), int(blk_off[r + 1])
        if b == a:
            continue
        if falls:
            v = rng.integers(1, 60, size=b - a)
        else:
            v = np.sort(rng.integers(1, 60, size=b - a))
        cold = int(rng.integers(0, b - a + 1))  # cold blocks form a suffix of the request
        v = v.astype(np.uint64)
        if cold < b - a:
            v[cold:] = NONE
        dist[a:b] = v
    caps = sorted(set(int(c) for c in rng.integers(1, 80, size=int(rng.integers(1, 12)))))
    B = int(rng.choice([1, 2, 16]))
    for kind in (0, 1, 2):
        h, s, t = _curves_by_definition(dist, blk_off, caps, B, kind)
        g = _gpu_curves(dist, blk_off, caps, B, kind)
        assert g["hits"] == h and g["saved"] == s and g["total_cost"] == t, (kind, seed, falls)


def test_long_requests_across_tiles():
    """Requests far longer than one 4,096-access tile, with a fall late in
    one of them (the running max must carry across tiles)."""
    rng = np.random.default_rng(7)
    lens = [9000, 5, 13000, 1, 4100]
    blk_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    n = int(blk_off[-1])
    dist = np.sort(rng.integers(1, 5000, size=n)).astype(np.uint64)
    for r in range(len(lens)):
        a, b = int(blk_off[r]), int(blk_off[r + 1])
        dist[a:b] = np.sort(dist[a:b])
    caps = [1, 10, 100, 1000, 2500, 4999]
    h, s, t = _curves_by_definition(dist, blk_off, caps, 16, 1)
    g = _gpu_curves(dist, blk_off, caps, 16, 1)
    assert g["hits"] == h and g["saved"] == s and g["total_cost"] == t
    a = int(blk_off[2])
    dist[a + 8000] = 1  # a fall deep inside the third request
    h, s, t = _curves_by_definition(dist, blk_off, caps, 16, 1)
    g = _gpu_curves(dist, blk_off, caps, 16, 1)
    assert g["hits"] == h and g["saved"] == s and g["total_cost"] == t


def test_many_short_requests_in_one_tile():
    """More requests in one tile than its offset table holds."""
    rng = np.random.default_rng(3)
    lens = rng.integers(0, 4, size=3000)
    blk_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    n = int(blk_off[-1])
    dist = rng.integers(1, 30, size=n).astype(np.uint64)
    caps = [1, 2, 5, 10, 20, 29]
    for kind in (0, 1):
        h, s, t = _curves_by_definition(dist, blk_off, caps, 4, kind)
        g = _gpu_curves(dist, blk_off, caps, 4, kind)
        assert g["hits"] == h and g["saved"] == s and g["total_cost"] == t
