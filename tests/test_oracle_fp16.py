"""Pins for the oracle's binary16 codec and single ops (paper Sec. 3: IEEE-754
binary16, roundTiesToEven).  The oracle is checked against the format's
definition and against numpy's independent float16 implementation."""
import numpy as np

ALL = np.arange(65536, dtype=np.uint16)


def test_decode_matches_numpy_all_patterns(orc):
    mine = orc.f16_to_f64(ALL)
    ref = ALL.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(mine), nan)
    assert np.array_equal(mine[~nan], ref[~nan])
    # signed zeros
    assert np.signbit(mine[0x8000]) and not np.signbit(mine[0x0000])


def test_decode_definition_spot_values(orc):
    d = orc.f16_to_f64(np.array([0x0001, 0x03FF, 0x0400, 0x3C00, 0x3C01, 0x7BFF, 0x7C00, 0xFC00,
                                 0xC000, 0x3555], np.uint16))
    assert d[0] == 2.0 ** -24                         # smallest subnormal
    assert d[1] == 1023 * 2.0 ** -24                  # largest subnormal
    assert d[2] == 2.0 ** -14                         # smallest normal
    assert d[3] == 1.0 and d[4] == 1.0 + 2.0 ** -10
    assert d[5] == 65504.0
    assert d[6] == np.inf and d[7] == -np.inf
    assert d[8] == -2.0
    assert d[9] == (1024 + 0x155) * 2.0 ** (0xD - 25)


def test_roundtrip_all_finite_patterns(orc):
    vals = orc.f16_to_f64(ALL)
    finite = ~np.isnan(vals)
    back = orc.f64_to_f16(vals[finite])
    assert np.array_equal(back, ALL[finite])


def test_midpoints_tie_to_even(orc):
    # every pair of adjacent positive finite binary16 values (incl. subnormals)
    lo = np.arange(0x0000, 0x7BFF, dtype=np.uint16)
    hi = lo + 1
    a, b = orc.f16_to_f64(lo), orc.f16_to_f64(hi)
    mid = (a + b) / 2  # exact in binary64
    got = orc.f64_to_f16(mid)
    even = np.where(lo % 2 == 0, lo, hi)
    assert np.array_equal(got, even)
    # just off the midpoint goes to the nearer neighbour
    eps = (b - a) * 2.0 ** -20
    assert np.array_equal(orc.f64_to_f16(mid - eps), lo)
    assert np.array_equal(orc.f64_to_f16(mid + eps), hi)
    # negative side mirrors
    assert np.array_equal(orc.f64_to_f16(-mid), even | 0x8000)


def test_overflow_and_underflow_edges(orc):
    f = lambda v: int(orc.f64_to_f16(np.array([v]))[0])
    assert f(65504.0) == 0x7BFF
    assert f(65519.99) == 0x7BFF
    assert f(65520.0) == 0x7C00          # tie rounds to even -> overflow
    assert f(-1e9) == 0xFC00
    assert f(2.0 ** -25) == 0x0000       # tie between 0 and 2^-24: even is 0
    assert f(2.0 ** -25 * 1.0000001) == 0x0001
    assert f(3 * 2.0 ** -25) == 0x0002   # tie between 1 and 2 quanta: even is 2
    assert f(-2.0 ** -30) == 0x8000      # keeps the sign of zero
    assert f(float("nan")) & 0x7C00 == 0x7C00 and f(float("nan")) & 0x3FF


def test_encode_matches_numpy_random(orc):
    rng = np.random.default_rng(1911)
    mag = np.exp2(rng.uniform(-30, 17, 2_000_000))
    x = mag * np.where(rng.random(mag.size) < 0.5, -1.0, 1.0)
    mine = orc.f64_to_f16(x)
    ref = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(mine, ref)


def _interesting_f16(rng, n):
    pats = rng.integers(0, 0x7C00, n, dtype=np.uint16)       # finite magnitudes
    pats |= (rng.random(n) < 0.5).astype(np.uint16) << 15    # random signs
    return pats


def test_single_ops_match_numpy(orc):
    rng = np.random.default_rng(7384)
    n = 20000
    a, b = _interesting_f16(rng, n), _interesting_f16(rng, n)
    fa, fb = a.view(np.float16), b.view(np.float16)
    with np.errstate(all="ignore"):
        ref_add = (fa + fb).view(np.uint16)
        ref_sub = (fa - fb).view(np.uint16)
        ref_mul = (fa * fb).view(np.uint16)
    got_add = np.array([orc.h_add(int(x), int(y)) for x, y in zip(a, b)], np.uint16)
    got_sub = np.array([orc.h_sub(int(x), int(y)) for x, y in zip(a, b)], np.uint16)
    got_mul = np.array([orc.h_mul(int(x), int(y)) for x, y in zip(a, b)], np.uint16)
    assert np.array_equal(got_add, ref_add)
    assert np.array_equal(got_sub, ref_sub)
    assert np.array_equal(got_mul, ref_mul)


def test_signed_zero_rules(orc):
    assert orc.h_add(0x0000, 0x8000) == 0x0000   # +0 + -0 = +0
    assert orc.h_add(0x8000, 0x8000) == 0x8000   # -0 + -0 = -0
    assert orc.h_sub(0x8000, 0x8000) == 0x0000   # -0 - -0 = +0
    assert orc.h_sub(0x8000, 0x0000) == 0x8000   # -0 - +0 = -0
    assert orc.h_mul(0x8000, 0x3C00) == 0x8000   # -0 * 1 = -0
