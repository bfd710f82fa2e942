"""Pins of the oracle's quiescence guard (count of nonzero words) against
numpy's count_nonzero of the bit patterns."""
import numpy as np

import oracle


def test_count_nonzero_matches_numpy():
    rng = np.random.default_rng(21)
    for n in (0, 1, 7, 1000, 65537):
        h = rng.integers(0, 2**16, size=n, dtype=np.uint64).astype(np.uint16)
        h[rng.random(n) < 0.5] = 0
        assert oracle.count_nonzero(h) == int(np.count_nonzero(h))
        u = rng.integers(0, 2**32, size=n, dtype=np.uint64).astype(np.uint32)
        u[rng.random(n) < 0.3] = 0
        assert oracle.count_nonzero(u) == int(np.count_nonzero(u))
        assert oracle.count_nonzero(u.view(np.float32)) == int(np.count_nonzero(u))


def test_negative_zero_counts():
    assert oracle.count_nonzero(np.array([0, 0x8000, 0], np.uint16)) == 1
    assert oracle.count_nonzero(np.array([0.0, -0.0], np.float32)) == 1
