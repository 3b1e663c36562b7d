"""The random read-modify-write probe (a measurement hook): every slot it
claims is one that some probe's seeded index names, holds that probe's
number and the seed, and the claimed slots are exactly the distinct indices
the probes name."""
import numpy as np
import pytest
import torch

import paper_2609_28870_gb300 as ptc

pytestmark = pytest.mark.gpu

GOLDEN = np.uint64(0x9E3779B97F4A7C15)


def splitmix64_at(seed, n):
    """SplitMix64 (Steele, Lea and Flood 2014) output n of a stream seeded with `seed`."""
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (n.astype(np.uint64) + np.uint64(1)) * GOLDEN
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


@pytest.mark.parametrize("log2_slots,probes,seed", [(12, 3000, 7), (16, 50000, 123456789), (10, 5000, 0)])
def test_probe_claims_the_named_slots(log2_slots, probes, seed):
    L = ptc.lib()
    slots = 1 << log2_slots
    table = torch.full((slots, 2), -1, dtype=torch.int64, device="cuda")
    sink = torch.zeros(1, dtype=torch.int64, device="cuda")
    s = torch.cuda.current_stream()
    assert L.ptc_probe_random_rmw(table.data_ptr(), slots, probes, seed, sink.data_ptr(), s.cuda_stream) == 0
    torch.cuda.synchronize()
    t = table.cpu().numpy().view(np.uint64)
    named = splitmix64_at(seed, np.arange(probes)) & np.uint64(slots - 1)
    claimed = np.nonzero(t[:, 0] != np.uint64(2**64 - 1))[0]
    assert np.array_equal(np.sort(claimed.astype(np.uint64)), np.unique(named))
    # each claimed slot holds the number of a probe that names it, and the seed
    who = t[claimed, 0]
    assert np.all(who < probes)
    assert np.array_equal(named[who.astype(np.int64)], claimed.astype(np.uint64))
    assert np.all(t[claimed, 1] == np.uint64(seed))
