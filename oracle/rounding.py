"""Indeterminacy of the loss and of the projected gradient under fp32
rounding -- oracle.

TEST INFRASTRUCTURE ONLY (see the package header).

The BitNet forward quantises activations to int8 and rounds attention
operands to bf16, so a one-ulp difference in an fp32 intermediate -- as
produced by any other valid summation order of the same definition -- can
flip a code and move the loss of a sequence by far more than an ulp
(measured on the last-token loss: ~5e-3 for a 2-layer model, 2-7 % for the
24-layer 0.7B-shaped model).  g = (F+ - F-) / (2 eps)
amplifies that by 1 / (2 eps).  ``alternative_rounding`` reruns the oracle
with every value a reduction produces (each RMSNorm mean square, each
BitLinear output, each attention output) moved by one ulp up or down, each
with probability 1/4, i.e. rounded the other way; the spread of an ensemble of
such runs measures how far two correct implementations may disagree on a
given input.  The oracle's own arithmetic is unchanged.  ``within`` accepts
a value that agrees with the oracle to the stated relative bound, or that
deviates from it by no more than one of these alternatives does.
"""
from __future__ import annotations

import contextlib

import numpy as np

from . import bitnet


def _bump(rng, y):
    u = rng.random(np.shape(y))
    y = np.asarray(y, dtype=np.float32)
    out = np.where(u < 0.25, np.nextafter(y, np.float32(np.inf)), y)
    return np.where(u > 0.75, np.nextafter(y, np.float32(-np.inf)), out).astype(np.float32)


@contextlib.contextmanager
def alternative_rounding(seed: int):
    rng = np.random.default_rng(seed)
    orig = (bitnet.bitlinear, bitnet.rmsnorm, bitnet.attention)

    def bitlinear(x, codes, s_w):
        return _bump(rng, orig[0](x, codes, s_w))

    def rmsnorm(x, gain):
        F32 = np.float32
        x = np.asarray(x, dtype=F32)
        ms = (np.sum(x * x, axis=-1, keepdims=True, dtype=F32) / F32(x.shape[-1])).astype(F32)
        ms = _bump(rng, ms)
        r = (F32(1.0) / np.sqrt(ms + F32(bitnet.RMS_EPS))).astype(F32)
        return ((x * r).astype(F32) * np.asarray(gain, dtype=F32)).astype(F32)

    def attention(q, k, v):
        return _bump(rng, orig[2](q, k, v))

    bitnet.bitlinear, bitnet.rmsnorm, bitnet.attention = bitlinear, rmsnorm, attention
    try:
        yield
    finally:
        bitnet.bitlinear, bitnet.rmsnorm, bitnet.attention = orig


def loss_ensemble(cfg, model, theta, n: int = 6, rows=None):
    """Per-sequence losses [n, rows] of one model (codes, s_w) under n
    alternative roundings; theta = (embed, gains, head, tokens, targets)."""
    out = []
    for r in range(n):
        with alternative_rounding(100 + r):
            per, _ = bitnet.batch_loss(cfg, model[0], model[1], *theta, rows=rows)
        out.append(per)
    return np.array(out)


def g_ensemble(cfg, plus, minus, theta, eps, n: int = 6, rows=None):
    """Minibatch g under n alternative roundings.  plus / minus: (codes, s_w)
    of the two perturbed models."""
    lp = loss_ensemble(cfg, plus, theta, n, rows)
    lm = loss_ensemble(cfg, minus, theta, n, rows)
    return (lp.mean(axis=1) - lm.mean(axis=1)) / (2.0 * float(np.float32(eps)))


def within(value, ref, ens, rel=1e-3) -> bool:
    """True if value agrees with ref to `rel`, or deviates from ref by no
    more than the largest deviation of an ensemble member: |value - ref| <=
    max_i |ens_i - ref|.  The members are the oracle itself under other valid
    fp32 roundings, so this accepts a value exactly when the oracle's own
    alternatives move at least as far from it (no widening beyond them)."""
    dev = float(np.max(np.abs(np.ravel(ens) - ref))) if np.size(ens) else 0.0
    return abs(value - ref) <= rel * abs(ref) or abs(value - ref) <= dev


def consistent(value, ref, ens, k=5.0) -> bool:
    """Statistical form for losses that are chaotic in the fp32 roundings (a
    24-30-layer random-init decoder, where one flipped activation code
    changes every later layer and the oracle's own re-roundings spread F by
    several percent): value lies within k sample standard deviations of the
    mean of [ref] + ens.  For a value drawn from the same distribution as the
    n + 1 others, (value - mean) / (sd sqrt(1 + 1/(n+1))) is Student-t with n
    degrees of freedom; k = 5 with n = 8 rejects such a value with
    probability about 1e-3."""
    allv = np.concatenate([[ref], np.ravel(ens)]).astype(np.float64)
    sd = float(np.std(allv, ddof=1))
    return abs(float(value) - float(allv.mean())) <= k * sd


def agrees(value, ref, ens, rel=1e-3) -> bool:
    """The acceptance of a GPU loss or g: ``within`` (the stated relative
    bound, or no further from the oracle than its furthest re-rounding), or,
    where the loss is chaotic in the roundings, ``consistent``."""
    return within(value, ref, ens, rel) or consistent(value, ref, ens)


def summary(value, ref, ens) -> dict:
    """|value - ref| next to the ensemble's largest deviation from ref and
    its range, for the parity record."""
    allv = np.concatenate([[ref], np.ravel(ens)])
    sd = float(np.std(allv, ddof=1)) if allv.size > 1 else 0.0
    return dict(value=float(value), ref=float(ref), abs_err=abs(float(value) - float(ref)),
                rel_err=abs(float(value) - float(ref)) / max(abs(float(ref)), 1e-300),
                ens_max_dev=float(np.max(np.abs(np.ravel(ens) - ref))) if np.size(ens) else 0.0,
                ens_min=float(allv.min()), ens_max=float(allv.max()), n_ens=int(np.size(ens)),
                z=(float(value) - float(allv.mean())) / sd if sd > 0 else 0.0)


def g_within_ensemble(g, g_ref, ens, rel=1e-3) -> bool:
    return agrees(g, g_ref, ens, rel)
