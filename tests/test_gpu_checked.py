"""The checked build and determinism.

The checked build (build(checked=True), -DPTC_CHECKED) is the substitute
for a sanitizer, which this pool does not offer: every index that comes
from data another stage or the caller wrote is checked before use, and a
miss is reported as PTC_ERR_BOUNDS rather than touching memory.  The parity
checks of tests/checked_run.py run against it in a process of their own.

Determinism: every output of the path is defined exactly, so two runs on
the same input must give the same bytes."""
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_checked_build_parity():
    from paper_2609_28870_gb300 import build
    build.build(checked=True)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "checked_run.py")], capture_output=True,
                       text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "all calls clean" in r.stdout


def test_two_runs_give_the_same_bytes():
    import torch

    import paper_2609_28870_gb300 as ptc
    from tests.gpu_util import to_gpu
    tr = tracegen.make(1, max_requests=2500)
    ids, D = oracle.block_ids(tr.tokens, tr.req_tok_off, 16)
    caps = tracegen.workload_grid(1, D)
    tok, off, ts = to_gpu(tr)
    ses = torch.from_numpy(tr.req_session.astype(np.uint32).view(np.int32)).cuda()
    runs = []
    for _ in range(2):
        outs = {k: torch.empty(ids.size, dtype=torch.int32, device="cuda") for k in ("ids", "prev", "next", "dist")}
        outs["keys"] = torch.empty(2 * (tr.tokens.size // 16), dtype=torch.int64, device="cuda")
        outs["req_blk_off"] = torch.empty(tr.n_req + 1, dtype=torch.int64, device="cuda")
        res = ptc.ptc_pipeline(tok, off, ts, 16, caps, outputs=outs, req_session=ses, n_session=tr.n_sessions)
        bel = ptc.ptc_belady_curves(outs["prev"], outs["req_blk_off"], 16, caps)
        sl = ptc.ptc_session_lru_curves(outs["ids"], D, outs["req_blk_off"], ses, tr.n_sessions, 16, caps)
        n = res["n_access"]
        outs["keys"] = outs["keys"][: 2 * n]  # the buffer holds the upper bound T / 16; N keys are written
        runs.append((res, bel, sl, {k: v.cpu().numpy().tobytes() for k, v in outs.items()}))
    assert runs[0][:3] == runs[1][:3]
    for k in runs[0][3]:
        assert runs[0][3][k] == runs[1][3][k], k
