"""Pins of the oracle's counter-based random stream (CPU only)."""
import os

import numpy as np
from scipy import stats

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            w = [int(t, 16) for t in line.split()]
            rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_philox_known_answers(orc):
    kat = _kat()
    assert len(kat) == 3
    for ctr, key, want in kat:
        assert list(orc.philox(ctr, key)) == want


def test_uniform_layout_and_grid(orc):
    # U(draw) uses word draw%4 of the block with counter {draw/4, node, batch, purpose}
    seed = 0x1234_5678_9ABC_DEF0
    for purpose, b, node in [(0, 0, 0), (1, 3, 17), (3, 65535, 1023)]:
        for draw in [0, 1, 2, 3, 4, 151935]:
            u = orc.uniform(seed, purpose, b, node, draw)
            w = orc.philox([draw >> 2, node, b, purpose], [seed & 0xFFFFFFFF, seed >> 32])[draw & 3]
            assert u == ((int(w) >> 8) + 0.5) / 2.0**24
            k = u * 2.0**24 - 0.5
            assert k == int(k) and 0 <= k < 2**24
            assert 0.0 < u < 1.0


def test_uniform_is_uniform(orc):
    us = np.array([orc.uniform(7, 1, 0, 5, d) for d in range(20000)])
    assert stats.kstest(us, "uniform").pvalue > 1e-3
    # different purposes / nodes / batches give different streams
    a = [orc.uniform(7, 1, 0, 5, d) for d in range(64)]
    b = [orc.uniform(7, 1, 0, 6, d) for d in range(64)]
    c = [orc.uniform(7, 2, 0, 5, d) for d in range(64)]
    d = [orc.uniform(7, 1, 1, 5, d) for d in range(64)]
    assert a != b and a != c and a != d
