"""The input generator: determinism, shapes, and its real-valued helpers."""
import math

import numpy as np

import tracegen


def test_deterministic_and_sorted():
    a = tracegen.make(0, max_requests=300)
    b = tracegen.make(0, max_requests=300, threads=3)
    assert np.array_equal(a.tokens, b.tokens)
    assert np.array_equal(a.req_tok_off, b.req_tok_off)
    assert np.all(np.diff(a.req_ts_us) >= 0)
    assert a.tokens.max() < 151936
    c = tracegen.make(0, seed=5, max_requests=300)
    assert not np.array_equal(a.tokens[:1000], c.tokens[:1000])


def test_workload_scale():
    """Session counts are set so the tiny trace has ~2,000 requests and the
    chat / agentic / mixed traces ~150M / ~2B / ~10B tokens (within 10%)."""
    r0, t0, s0 = tracegen.sizes(0)
    assert 1800 <= r0 <= 2200 and s0 == 444
    _, t1, _ = tracegen.sizes(1)
    assert 135e6 <= t1 <= 165e6
    _, t2, _ = tracegen.sizes(2)
    assert 1.8e9 <= t2 <= 2.2e9
    _, t3, _ = tracegen.sizes(3)
    assert 9e9 <= t3 <= 11e9


def test_agentic_cap_and_prefix_growth():
    tr = tracegen.make(2, sessions=40)
    lens = np.diff(tr.req_tok_off)
    assert lens.max() <= 131072
    # each request of a session extends the previous one until truncation
    last = {}
    grow = 0
    for r in range(tr.n_req):
        s = int(tr.req_session[r])
        a, b = int(tr.req_tok_off[r]), int(tr.req_tok_off[r + 1])
        if s in last:
            pa, pb = last[s]
            n = min(pb - pa, b - a)
            if np.array_equal(tr.tokens[pa:pa + n], tr.tokens[a:a + n]):
                grow += 1
        last[s] = (a, b)
    assert grow > 0


def test_det_functions_close_to_libm():
    lib = tracegen._load()
    for x in [1e-300, 1e-9, 0.3, 0.5, 0.7071, 1.0, 2.0, 10.0, 12345.678, 1e300]:
        assert abs(lib.tg_det_log(x) - math.log(x)) <= 1e-12 * max(1.0, abs(math.log(x)))
    for x in [-700.0, -30.0, -1.0, 0.0, 1e-5, 0.5, 1.0, 20.0, 700.0]:
        assert abs(lib.tg_det_exp(x) - math.exp(x)) <= 1e-12 * math.exp(x)
    for x in np.linspace(0, 4 * math.pi, 97):
        assert abs(lib.tg_det_cos(float(x)) - math.cos(x)) <= 1e-12


def test_capacity_grid():
    g = tracegen.capacity_grid(64, 135640, 16)
    assert g[0] == 64 and g[-1] == 135640 and np.all(np.diff(g.astype(np.int64)) > 0) and g.size == 16
    g = tracegen.capacity_grid(1, 3, 8)
    assert g.tolist() == list(range(1, 9))
