"""Pins for the oracle's Philox4x32-10 and draw layout."""
import os

import numpy as np

from oracle import philox

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        w = [int(x, 16) for x in line.split()]
        rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_known_answer_vectors():
    rows = _kat()
    assert len(rows) == 3
    for ctr, key, want in rows:
        assert list(philox.philox4x32_10(ctr, key)) == want


def test_vectorised_matches_scalar():
    rows = _kat()
    for ctr, key, want in rows:
        out = philox.philox4x32_10_np(*[np.array([c], dtype=np.uint64) for c in ctr],
                                      np.array([key[0]], dtype=np.uint64), np.array([key[1]], dtype=np.uint64))
        assert [int(o[0]) for o in out] == want
    b = np.arange(50)
    for draw in (0, 16, 32, 33):
        v = philox.uniforms_np(12345678901, b, 3, draw)
        s = [philox.uniform(12345678901, int(x), 3, draw) for x in b]
        assert np.array_equal(v, np.array(s))


def test_uniform_grid_and_range():
    u = philox.uniforms_np(7, np.arange(200000), 1, 16)
    assert u.min() >= 0.0 and u.max() < 1.0
    k = u * 2.0 ** 24
    assert np.array_equal(k, np.floor(k))
    # mean and a coarse histogram of a correct generator
    assert abs(u.mean() - 0.5) < 5 * np.sqrt(1 / 12 / len(u))
    h = np.histogram(u, bins=16, range=(0, 1))[0] / len(u)
    assert np.abs(h - 1 / 16).max() < 5 * np.sqrt(1 / 16 / len(u))


def test_draws_are_keyed_by_every_field():
    base = philox.uniform(1, 2, 3, 4)
    assert philox.uniform(1, 2, 3, 5) != base
    assert philox.uniform(1, 2, 4, 4) != base
    assert philox.uniform(1, 3, 3, 4) != base
    assert philox.uniform(2, 2, 3, 4) != base
    assert philox.uniform(1 + (1 << 32), 2, 3, 4) != base
