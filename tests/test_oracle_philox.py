"""Pins of the oracle's perturbation generator: Philox-4x32-10 against the
authors' published known-answer vectors, Box-Muller against exact identities
and the normal distribution.  CPU only."""
import os

import numpy as np
import pytest

from oracle import philox

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            rows.append([int(x, 16) for x in line.split()])
    return rows


def test_philox_known_answers():
    rows = _kat()
    assert len(rows) == 3
    for r in rows:
        out = philox.philox4x32_10(*r[:6])
        assert [int(o) for o in out] == r[6:]


def test_counter_layout_and_lanes():
    seed = 0x1234_5678_9ABC_DEF0
    idx = np.arange(64, dtype=np.uint64)
    words = philox.raw_words(seed, idx)
    for i in (0, 5, 63):
        g = i // 4
        out = philox.philox4x32_10(g, 0, 0, 0, seed & 0xFFFFFFFF, seed >> 32)
        assert int(words[i]) == int(out[i % 4])
    # a large index uses the high counter word
    big = np.array([(1 << 34) + 6], dtype=np.uint64)
    out = philox.philox4x32_10(((1 << 34) + 6) // 4 & 0xFFFFFFFF, ((1 << 34) + 6) // 4 >> 32, 0, 0,
                               seed & 0xFFFFFFFF, seed >> 32)
    assert int(philox.raw_words(seed, big)[0]) == int(out[2])


def test_uniform_is_exact_and_open():
    u = np.array([0, 1 << 9, 0xFFFFFFFF, 0x80000000], dtype=np.uint32)
    x = philox.uniform(u)
    assert x[0] == np.float32(2.0 ** -24)
    assert x[1] == np.float32(3 * 2.0 ** -24)
    assert x[2] == np.float32(1.0 - 2.0 ** -24)
    assert x[3] == np.float32(0.5 + 2.0 ** -24)
    assert np.all((x > 0) & (x < 1))


def test_normal_moments_and_ks():
    stats = pytest.importorskip("scipy.stats")
    z = philox.normal(42, np.arange(1 << 20)).astype(np.float64)
    assert abs(z.mean()) < 5e-3
    assert abs(z.var() - 1.0) < 5e-3
    assert abs(((z - z.mean()) ** 4).mean() / z.var() ** 2 - 3.0) < 3e-2
    assert stats.kstest(z, "norm").pvalue > 1e-3
    assert abs(np.corrcoef(z[0::2], z[1::2])[0, 1]) < 5e-3


def test_box_muller_radius_and_angle_identities():
    seed = 77
    idx = np.arange(0, 4096, dtype=np.uint64)
    z = philox.normal(seed, idx).astype(np.float64)
    xa = philox.uniform(philox.raw_words(seed, idx[0::2])).astype(np.float64)
    xb = philox.uniform(philox.raw_words(seed, idx[1::2])).astype(np.float64)
    r2 = z[0::2] ** 2 + z[1::2] ** 2
    np.testing.assert_allclose(r2, -2.0 * np.log(xa), rtol=2e-6, atol=1e-6)
    ang = np.arctan2(z[1::2], z[0::2]) % (2 * np.pi)
    d = np.abs(ang - 2 * np.pi * xb)
    d = np.minimum(d, 2 * np.pi - d)
    assert np.all(d < 1e-4)


def test_z_depends_only_on_seed_and_index():
    idx = np.array([3, 1000, 17, 999999], dtype=np.uint64)
    full = philox.normal(5, np.arange(1000000, dtype=np.uint64))
    assert np.array_equal(philox.normal(5, idx), full[idx.astype(np.int64)])
    assert not np.array_equal(philox.normal(6, idx), philox.normal(5, idx))
