"""Pins of the oracle's appended-slot noise (Sec. 3.1: the new slot ~ N(0, I)).

Each test checks the oracle against something other than itself: published
Philox known-answer vectors, libm in float64, the exact Taylor coefficients,
and the Gaussian distribution.
"""
import os
from fractions import Fraction

import mpmath
import numpy as np
import pytest
from scipy import stats

from oracle import noise

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")

# every reachable uniform: odd multiples of 2^-24 in (0, 1)
_ALL_U = ((2 * np.arange(2 ** 23, dtype=np.int64) + 1).astype(np.float32) * np.float32(2.0 ** -24))


def test_philox_known_answers():
    rows = [ln.split() for ln in open(GOLDEN) if ln.strip() and not ln.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(t, 16) for t in r]
        out = noise.philox4x32_10(v[0:4], v[4:6])
        assert [int(o) for o in out] == v[6:10]


def test_philox_vectorised_matches_scalar():
    rng = np.random.default_rng(1)
    c = rng.integers(0, 2 ** 32, size=(4, 64), dtype=np.uint64)
    k = rng.integers(0, 2 ** 32, size=(2, 64), dtype=np.uint64)
    vec = noise.philox4x32_10(tuple(c), tuple(k))
    for i in range(64):
        sc = noise.philox4x32_10(tuple(int(x) for x in c[:, i]), tuple(int(x) for x in k[:, i]))
        assert [int(s) for s in sc] == [int(v[i]) for v in vec]


def test_uniform_map_is_open_interval_and_exact():
    u = noise.bits_to_uniform(np.array([0, 511, 512, 0xFFFFFFFF], dtype=np.uint32))
    assert u[0] == np.float32(2.0 ** -24) and u[1] == u[0]
    assert u[2] == np.float32(3 * 2.0 ** -24)
    assert u[3] == np.float32(1 - 2.0 ** -24)
    assert np.all((u > 0) & (u < 1))


def _cr_f32(x) -> np.float32:
    """Correctly rounded float32 of an mpmath number."""
    fr = Fraction(int(mpmath.nint(x * mpmath.mpf(2) ** 160)), 2 ** 160)
    c = np.float32(float(x))
    cands = [np.nextafter(c, np.float32(-np.inf)), c, np.nextafter(c, np.float32(np.inf))]
    return min(cands, key=lambda v: abs(Fraction(float(v)) - fr))


def test_polynomial_constants_are_correctly_rounded():
    mpmath.mp.dps = 50
    hp = mpmath.pi / 2
    for i, n in enumerate((1, 3, 5, 7, 9)):
        assert noise.SIN_C[i] == _cr_f32((-1) ** i * hp ** n / mpmath.factorial(n))
    for i, n in enumerate((0, 2, 4, 6, 8, 10)):
        assert noise.COS_C[i] == _cr_f32((-1) ** i * hp ** n / mpmath.factorial(n))
    for c, n in ((noise.LN_C3, 3), (noise.LN_C5, 5), (noise.LN_C7, 7), (noise.LN_C9, 9)):
        assert c == _cr_f32(mpmath.mpf(1) / n)
    # LN2_HI has few enough bits that e * LN2_HI is exact for |e| <= 2^8
    hi_bits = int(np.array([noise.LN2_HI]).view(np.uint32)[0]) & 0x7FFFFF
    assert hi_bits & 0x1FF == 0
    assert noise.LN2_LO == _cr_f32(mpmath.log(2) - mpmath.mpf(float(noise.LN2_HI)))


def test_own_ln_within_3_ulp_of_libm_on_every_reachable_u():
    got = noise.ln_f32(_ALL_U).astype(np.float64)
    ref = np.log(_ALL_U.astype(np.float64))
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(got - ref) / ulp) <= 3.0


def test_own_sincos_within_2e7_of_libm_on_every_reachable_u():
    s, c = noise.sincos_2pi_f32(_ALL_U)
    ang = 2.0 * np.pi * _ALL_U.astype(np.float64)
    assert np.max(np.abs(s - np.sin(ang))) < 2e-7
    assert np.max(np.abs(c - np.cos(ang))) < 2e-7
    # exact special points
    s, c = noise.sincos_2pi_f32(np.array([0.0, 0.25, 0.5, 0.75, 1.0], np.float32))
    np.testing.assert_array_equal(s, np.array([0, 1, 0, -1, 0], np.float32))
    np.testing.assert_array_equal(np.abs(c), np.array([1, 0, 1, 0, 1], np.float32))


def test_box_muller_matches_float64_formula():
    rng = np.random.default_rng(5)
    ua = noise.bits_to_uniform(rng.integers(0, 2 ** 32, 200000, dtype=np.uint64).astype(np.uint32))
    ub = noise.bits_to_uniform(rng.integers(0, 2 ** 32, 200000, dtype=np.uint64).astype(np.uint32))
    z0, z1 = noise.box_muller(ua, ub)
    r = np.sqrt(-2.0 * np.log(ua.astype(np.float64)))
    ang = 2 * np.pi * ub.astype(np.float64)
    np.testing.assert_allclose(z0, r * np.cos(ang), rtol=0, atol=4e-6)
    np.testing.assert_allclose(z1, r * np.sin(ang), rtol=0, atol=4e-6)


def test_action_noise_is_standard_normal_and_independent():
    z = noise.action_noise(123, np.arange(40000, dtype=np.uint64), 32)   # 1.28e6 draws
    flat = z.ravel().astype(np.float64)
    assert abs(flat.mean()) < 5e-3 and abs(flat.var() - 1) < 5e-3
    assert stats.kstest(flat, "norm").pvalue > 1e-3
    # dims, actions and robots are uncorrelated
    corr = np.corrcoef(z[:, :8].T.astype(np.float64))
    assert np.max(np.abs(corr - np.eye(8))) < 0.03
    other = noise.action_noise(124, np.arange(40000, dtype=np.uint64), 32)
    assert abs(np.corrcoef(flat, other.ravel())[0, 1]) < 0.01


def test_action_noise_layout():
    # element 4g+i of action n is output i of the Philox block at counter (n, g)
    n = np.uint64(2 ** 33 + 7)
    seed = (5 << 32) | 9
    z = noise.action_noise(seed, n, 10)
    x = noise.philox4x32_10((int(n) & 0xFFFFFFFF, int(n) >> 32, 2, noise.NOISE_TAG), (9, 5))
    u = noise.bits_to_uniform(np.array(x, np.uint32))
    a, b = noise.box_muller(u[0:1], u[1:2])
    assert z[8] == a[0] and z[9] == b[0]
    assert z.shape == (10,)
