"""Ternary quantizer geometry (Sec. 3, "Ternary Quantization") -- oracle.

TEST INFRASTRUCTURE ONLY (see the package header).

* ``exact_abs_sum``  -- sum_i |w_i| of a float32 vector as an exact rational.
* ``absmean``        -- gamma = sum_i |w_i| / n (Sec. 3, text under Eq. 2).
  The paper fixes no precision or order for this sum; the reading used here
  is: the exact real sum, rounded once to float64, divided by n in float64,
  rounded to float32.  Being exact, it does not depend on summation order.
  Pinned against ``fractions.Fraction`` sums and closed forms.
* ``threshold``      -- tau = 0.5 (gamma + delta), delta = 1e-5 (the paper's
  example value), evaluated in float32.  ``weight_scale`` = gamma + delta,
  the dequantisation scale of the ternary weights (reading: the quantizer
  rounds w / (gamma + delta); the paper does not state the dequant scale).
* ``quantize``       -- Eq. 2 with strict inequalities: +1 if w > tau,
  -1 if w < -tau, else 0.  Pinned by brute force.
* ``distance``       -- Eq. 3, d_i = min(|w_i - tau|, |w_i + tau|), in float32.
  Pinned against the written-out min form, bit for bit.
* ``pack_codes``     -- 2-bit storage of ternary codes (Sec. 4, B_Q = 2/8
  byte): code q + 1 in bits 2*(i mod 16) of 32-bit word i // 16.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np

DELTA = np.float32(1e-5)


def _mant_exp(w: np.ndarray):
    """|w| = m * 2**(e - 150) with m < 2**24 an integer, e >= 1 (fp32)."""
    bits = np.ascontiguousarray(w, dtype=np.float32).view(np.uint32) & np.uint32(0x7FFFFFFF)
    e = (bits >> np.uint32(23)).astype(np.int64)
    m = (bits & np.uint32(0x7FFFFF)).astype(np.int64)
    m = np.where(e > 0, m | (1 << 23), m)
    e = np.maximum(e, 1)
    return m, e


def exact_abs_sum(w: np.ndarray) -> Fraction:
    """Exact rational value of sum_i |w_i| for float32 w (no rounding)."""
    w = np.asarray(w, dtype=np.float32).reshape(-1)
    if not np.all(np.isfinite(w)):
        raise ValueError("non-finite latent weight")
    total = 0
    chunk = 1 << 26  # keeps every per-exponent float64 partial below 2**53
    for s in range(0, w.size, chunk):
        m, e = _mant_exp(w[s:s + chunk])
        per_e = np.bincount(e, weights=m.astype(np.float64), minlength=256)
        for ee in np.nonzero(per_e)[0]:
            total += int(per_e[ee]) << int(ee)
    return Fraction(total, 1 << 150)


def absmean(w: np.ndarray) -> np.float32:
    """gamma = sum|w_i| / n: exact sum -> float64 -> / n (float64) -> float32."""
    n = int(np.asarray(w).size)
    if n == 0:
        raise ValueError("empty tensor")
    s_d = float(exact_abs_sum(w))  # correctly rounded to float64
    return np.float32(s_d / float(n))


def threshold(gamma: np.float32) -> np.float32:
    """tau = 0.5 * (gamma + delta) in float32."""
    return np.float32(np.float32(0.5) * np.float32(np.float32(gamma) + DELTA))


def weight_scale(gamma: np.float32) -> np.float32:
    """s_w = gamma + delta in float32 (= 2 tau exactly)."""
    return np.float32(np.float32(gamma) + DELTA)


def quantize(w: np.ndarray, tau: np.float32) -> np.ndarray:
    """Eq. 2: int8 codes in {-1, 0, +1}."""
    w = np.asarray(w, dtype=np.float32)
    tau = np.float32(tau)
    q = np.zeros(w.shape, dtype=np.int8)
    q[w > tau] = 1
    q[w < -tau] = -1
    return q


def distance(w: np.ndarray, tau: np.float32) -> np.ndarray:
    """Eq. 3 in float32: min(|w - tau|, |w + tau|)."""
    w = np.asarray(w, dtype=np.float32)
    tau = np.float32(tau)
    return np.minimum(np.abs(w - tau), np.abs(w + tau)).astype(np.float32)


def pack_codes(q: np.ndarray) -> np.ndarray:
    """Pack int8 codes (length a multiple of 16) into uint32 words."""
    q = np.asarray(q, dtype=np.int8).reshape(-1)
    if q.size % 16:
        raise ValueError("code count must be a multiple of 16")
    c = (q.astype(np.int64) + 1).reshape(-1, 16)
    shifts = 2 * np.arange(16, dtype=np.int64)
    return (c << shifts).sum(axis=1).astype(np.uint32)


def unpack_codes(words: np.ndarray) -> np.ndarray:
    """Inverse of pack_codes (code value 3 is reported as +2 to expose it)."""
    w = np.asarray(words, dtype=np.uint32).astype(np.int64).reshape(-1, 1)
    shifts = 2 * np.arange(16, dtype=np.int64)
    return (((w >> shifts) & 3) - 1).astype(np.int8).reshape(-1)
