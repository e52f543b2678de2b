"""Indeterminacy of the projected gradient under fp32 rounding -- oracle.

TEST INFRASTRUCTURE ONLY (see the package header).

The BitNet forward quantises activations to int8 (and, in this reading,
rounds attention operands to bf16), so a one-ulp difference in an fp32
intermediate -- as produced by any other valid summation order -- can flip
a code and move the loss by far more than an ulp.  g = (F+ - F-) / (2 eps)
divides that by 2 eps, so two correct fp32 implementations disagree on g.
``g_ensemble`` evaluates g under several alternative valid roundings (every
stored BitLinear output moved up by one ulp with probability 1/2, i.e.
rounded the other way) to measure that disagreement on a given input.
This does not change the oracle's arithmetic; it reruns it with perturbed
roundings.
"""
from __future__ import annotations

import contextlib

import numpy as np

from . import bitnet


@contextlib.contextmanager
def alternative_rounding(seed: int):
    orig = bitnet.bitlinear
    rng = np.random.default_rng(seed)

    def bl(x, codes, s_w):
        y = orig(x, codes, s_w)
        up = rng.random(y.shape) < 0.5
        return np.where(up, np.nextafter(y, np.float32(np.inf)), y).astype(np.float32)

    bitnet.bitlinear = bl
    try:
        yield
    finally:
        bitnet.bitlinear = orig


def g_ensemble(cfg, plus, minus, theta, eps, n: int = 6, rows=None):
    """g under n alternative roundings.  plus / minus: (codes, s_w) of the
    two perturbed models; theta: (embed, gains, head, tokens, targets)."""
    out = []
    for r in range(n):
        with alternative_rounding(100 + r):
            _, fp = bitnet.batch_loss(cfg, plus[0], plus[1], *theta, rows=rows)
            _, fm = bitnet.batch_loss(cfg, minus[0], minus[1], *theta, rows=rows)
        out.append((fp - fm) / (2.0 * float(np.float32(eps))))
    return np.array(out)


def g_within_ensemble(g, g_ref, ens, rel=1e-3) -> bool:
    """True if g agrees with g_ref to `rel`, or lies inside the ensemble's
    range [min, max] widened by its spread on both sides."""
    allg = np.concatenate([[g_ref], ens])
    spread = allg.max() - allg.min()
    return abs(g - g_ref) <= rel * abs(g_ref) or (allg.min() - spread <= g <= allg.max() + spread)
