"""Pins of the oracle's quantizer geometry (Sec. 3, Eqs. 2-3) against
exact rational arithmetic, an independent textbook formulation and
exhaustive bit patterns.  CPU only."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import ternary


def _frac_sum(w):
    return sum((Fraction(float(abs(x))) for x in np.asarray(w, dtype=np.float32)), Fraction(0))


def _adversarial(rng, n):
    """Random latents plus denormals, zeros, signed zeros and wide exponents."""
    w = (rng.standard_normal(n) * 0.02).astype(np.float32)
    w[::7] = np.float32(1e-40) * rng.integers(1, 50, size=w[::7].size)   # denormals
    w[3::11] = np.float32(0.0)
    w[5::13] = np.float32(-0.0)
    w[1::17] = (rng.standard_normal(w[1::17].size) * 1e4).astype(np.float32)
    w[2::19] = np.ldexp(1.0, rng.integers(-126, 100, size=w[2::19].size)).astype(np.float32)
    return w


@pytest.mark.parametrize("n", [1, 2, 17, 1000, 4097])
def test_exact_abs_sum_matches_rational_sum(n):
    rng = np.random.default_rng(n)
    w = _adversarial(rng, n)
    assert ternary.exact_abs_sum(w) == _frac_sum(w)


def test_absmean_is_order_independent_and_correctly_rounded():
    rng = np.random.default_rng(7)
    w = _adversarial(rng, 5000)
    g = ternary.absmean(w)
    for _ in range(3):
        assert ternary.absmean(rng.permutation(w)).view(np.uint32) == g.view(np.uint32)
    exact = _frac_sum(w) / len(w)
    # float32(float64(S) / n): within one float32 ulp of the exact mean
    err = abs(Fraction(float(g)) - exact)
    assert err <= Fraction(float(np.spacing(g)))


def test_absmean_closed_forms():
    c = np.float32(0.0123)
    assert ternary.absmean(np.full(999, c, np.float32)) == c
    assert ternary.absmean(np.array([c, -c], np.float32)) == c
    # [1, 2^-24]: the exact mean (1 + 2^-24) / 2 is a float64 that rounds
    # to 0.5 in float32 (ties to even)
    w = np.array([1.0, 2.0 ** -24], np.float32)
    assert ternary.absmean(w) == np.float32((1.0 + 2.0 ** -24) / 2.0)


def _round_half_away(x):
    return np.sign(x) * np.floor(np.abs(x) + 0.5)


def test_quantize_equals_textbook_absmean_rounding_except_ties():
    rng = np.random.default_rng(3)
    w = (rng.standard_normal(200000) * 0.02).astype(np.float32)
    gamma = ternary.absmean(w)
    tau = ternary.threshold(gamma)
    q = ternary.quantize(w, tau)
    # BitNet b1.58: clamp(round(w / (gamma + delta)), -1, 1), evaluated in float64
    ref = np.clip(_round_half_away(w.astype(np.float64) / (2.0 * float(tau))), -1, 1)
    ties = np.abs(np.abs(w.astype(np.float64)) - float(tau)) < 1e-12
    assert np.array_equal(q[~ties], ref[~ties].astype(np.int8))
    assert set(np.unique(q)) <= {-1, 0, 1}


def test_quantize_exhaustive_bit_patterns_around_tau():
    tau = np.float32(0.0079123)
    bits = tau.view(np.uint32).astype(np.int64)
    pats = np.arange(bits - 1000, bits + 1001).astype(np.uint32).view(np.float32)
    for sign in (1, -1):
        w = (sign * pats).astype(np.float32)
        q = ternary.quantize(w, tau)
        mag = pats.view(np.uint32).astype(np.int64)
        expect = np.where(mag > bits, sign, 0)   # strict inequality: w = +-tau -> 0
        assert np.array_equal(q, expect.astype(np.int8))


def test_threshold_and_scale():
    g = np.float32(0.016)
    tau = ternary.threshold(g)
    s = ternary.weight_scale(g)
    assert tau == np.float32(0.5) * s            # tau = s_w / 2 exactly
    assert abs(float(s) - (float(g) + 1e-5)) <= float(np.spacing(s))


def test_distance_min_form_equals_folded_form_bitwise():
    rng = np.random.default_rng(5)
    w = _adversarial(rng, 100000)
    tau = np.float32(0.0081)
    d = ternary.distance(w, tau)
    folded = np.abs(np.abs(w) - tau).astype(np.float32)
    assert np.array_equal(d.view(np.uint32), folded.view(np.uint32))
    assert np.array_equal(d, ternary.distance(-w, tau))
    assert ternary.distance(np.array([tau, -tau], np.float32), tau).tolist() == [0.0, 0.0]
    assert ternary.distance(np.array([0.0], np.float32), tau)[0] == tau


def test_pack_unpack_roundtrip_and_layout():
    rng = np.random.default_rng(9)
    q = rng.integers(-1, 2, size=16 * 33).astype(np.int8)
    words = ternary.pack_codes(q)
    assert words.dtype == np.uint32 and words.size == 33
    assert np.array_equal(ternary.unpack_codes(words), q)
    one = np.zeros(16, np.int8)
    one[0], one[15] = 1, -1
    # code+1 at bits 2*(i mod 16): element 0 -> 2 at bits 0-1, element 15 -> 0
    assert int(ternary.pack_codes(one)[0]) == (2 | sum(1 << (2 * i) for i in range(1, 15)))
