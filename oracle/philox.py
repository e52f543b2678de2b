"""Perturbation direction z of Algorithm 1 -- oracle.

TEST INFRASTRUCTURE ONLY (see the package header).

Algorithm 1 draws z ~ N(0, I_d) from a seed s_{t,k} and later re-draws the
same z from that seed for the update; the paper does not name a generator.
The reading used here is a counter-based stream keyed on (seed, global
weight index), so that z_i does not depend on the mask or on the order in
which weights are visited:

* Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as
  easy as 1, 2, 3", SC'11): key = (seed mod 2^32, seed >> 32); counter =
  (g mod 2^32, g >> 32, 0, 0) with g = i // 4; output word j = i mod 4.
  Pinned by the authors' published known-answer vectors.
* Uniform: x = (2 * (u >> 9) + 1) * 2^-24, an exact float32 in (0, 1).
* Box-Muller (1958) on the word pairs (0, 1) and (2, 3):
  r = sqrt(-2 ln x_a), z_a = r cos(2 pi x_b), z_b = r sin(2 pi x_b),
  evaluated in float64 and rounded to float32.  Pinned by moments, a
  Kolmogorov-Smirnov test and exact special values.
"""
from __future__ import annotations

import numpy as np

M0 = np.uint64(0xD2511F53)
M1 = np.uint64(0xCD9E8D57)
W0 = np.uint64(0x9E3779B9)
W1 = np.uint64(0xBB67AE85)
MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Ten Philox-4x32 rounds; arguments are arrays of 32-bit values."""
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & MASK32 for c in (c0, c1, c2, c3))
    k0 = np.asarray(k0, dtype=np.uint64) & MASK32
    k1 = np.asarray(k1, dtype=np.uint64) & MASK32
    for _ in range(10):
        p0 = M0 * c0
        p1 = M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ k0), lo1, (hi0 ^ c3 ^ k1), lo0
        k0 = (k0 + W0) & MASK32
        k1 = (k1 + W1) & MASK32
    return c0, c1, c2, c3


def raw_words(seed: int, idx: np.ndarray) -> np.ndarray:
    """The 32-bit Philox word that belongs to each global index."""
    idx = np.asarray(idx, dtype=np.uint64)
    g = idx >> np.uint64(2)
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    k0 = np.uint64(seed & 0xFFFFFFFF)
    k1 = np.uint64(seed >> 32)
    out = philox4x32_10(g & MASK32, g >> np.uint64(32), np.zeros_like(g), np.zeros_like(g), k0, k1)
    lane = (idx & np.uint64(3)).astype(np.int64)
    words = np.stack(out, axis=0)
    return words[lane, np.arange(idx.size)].astype(np.uint32)


def uniform(u: np.ndarray) -> np.ndarray:
    """Exact float32 uniform in (0, 1) from a 32-bit word."""
    u = np.asarray(u, dtype=np.uint64)
    return ((((u >> np.uint64(9)) << np.uint64(1)) | np.uint64(1)).astype(np.float64)
            * 2.0 ** -24).astype(np.float32)


def normal(seed: int, idx) -> np.ndarray:
    """z_i for the given global indices, float32."""
    idx = np.asarray(idx, dtype=np.uint64).reshape(-1)
    base = (idx >> np.uint64(1)) << np.uint64(1)          # first index of the pair
    ua = uniform(raw_words(seed, base)).astype(np.float64)
    ub = uniform(raw_words(seed, base + np.uint64(1))).astype(np.float64)
    r = np.sqrt(-2.0 * np.log(ua))
    theta = 2.0 * np.pi * ub
    first = (idx & np.uint64(1)) == 0
    z = np.where(first, r * np.cos(theta), r * np.sin(theta))
    return z.astype(np.float32)
