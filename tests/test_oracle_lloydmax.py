"""Pins for the Lloyd-Max codebook and group quantizer (CPU only).

The codebook is checked against what fixes it independently of the code that
computes it: the closed form at one bit (levels +-sqrt(2/pi), MSE 1 - 2/pi),
Max's published 2-bit levels, the exact MSE column of Table 8 (App. F), a
Monte-Carlo estimate of the MSE, and the fact that no uniform quantizer of
N(0, 1) does better. The group quantizer is checked against brute-force
nearest-level search.
"""
import math
import os

import numpy as np
import pytest

from oracle import lloydmax as lm

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def table8():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "table8_lloydmax.txt"))
            if l.strip() and not l.startswith("#")]
    return {int(r[0]): float(r[1]) for r in rows}


def test_one_bit_closed_form():
    lev, D = lm.design(1)
    a = math.sqrt(2.0 / math.pi)                  # E|X| of N(0, 1)
    np.testing.assert_allclose(lev, [-a, a], rtol=1e-14)
    assert D == pytest.approx(1.0 - 2.0 / math.pi, rel=1e-13)


def test_two_bit_levels_match_max_1960():
    # Max (1960), Table I, N = 4: outputs 0.4528, 1.510
    lev, _ = lm.design(2)
    np.testing.assert_allclose(lev, [-1.510, -0.4528, 0.4528, 1.510], atol=6e-4)


@pytest.mark.parametrize("b", [1, 2, 3, 4])
def test_table8_exact_mse(b):
    # the printed exact D(b) at b = 1..4 is D rounded to four significant digits
    _, D = lm.design(b)
    printed = table8()[b]
    half_unit = 0.5 * 10.0 ** (math.floor(math.log10(printed)) - 3)
    assert abs(D - printed) <= half_unit


@pytest.mark.parametrize("b", [5, 6])
def test_table8_tail_is_not_below_the_optimum(b):
    # Table 8 prints 2.512e-03 and 7.647e-04 at 5 and 6 bits; the converged
    # quantizer reaches 2.5047e-03 and 6.442e-04. An optimal quantizer can only
    # be at or below any printed quantizer's MSE, which these are.
    _, D = lm.design(b)
    assert D <= table8()[b]
    assert D == pytest.approx(table8()[b], rel=0.2)


@pytest.mark.parametrize("b", range(1, 9))
def test_fixed_point_symmetry_and_monte_carlo(b):
    lev, D = lm.design(b)
    t, p, c = lm._centroids(lev)
    assert np.all(np.diff(lev) > 0)
    np.testing.assert_allclose(lev, -lev[::-1], atol=0)
    assert np.max(np.abs(lev - c)) < 1e-10          # both Lloyd-Max conditions hold
    x = np.random.default_rng(100 + b).standard_normal(2_000_000)
    idx = np.searchsorted(0.5 * (lev[:-1] + lev[1:]), x, side="right")
    mc = np.mean((x - lev[idx]) ** 2)
    assert mc == pytest.approx(D, rel=0.01)


@pytest.mark.parametrize("b", [1, 2, 3, 4, 5])
def test_beats_every_uniform_quantizer(b):
    # the best uniform (mid-rise, n = 2^b levels) quantizer of N(0, 1) by a
    # fine search over the step: Lloyd-Max must not be worse
    from scipy.special import ndtr
    n = 2 ** b
    _, D = lm.design(b)

    def uniform_mse(step):
        lev = (np.arange(n) - (n - 1) / 2) * step
        t = np.concatenate([[-np.inf], 0.5 * (lev[:-1] + lev[1:]), [np.inf]])
        p = ndtr(t[1:]) - ndtr(t[:-1])
        phi = lambda z: np.where(np.isfinite(z), np.exp(-0.5 * np.where(np.isfinite(z), z, 0) ** 2), 0) / math.sqrt(2 * math.pi)
        m1 = phi(t[:-1]) - phi(t[1:])                  # E[X; cell]
        tz = np.where(np.isfinite(t), t, 0.0)
        m2 = p + tz[:-1] * phi(t[:-1]) - tz[1:] * phi(t[1:])   # E[X^2; cell]
        return float(np.sum(m2 - 2 * lev * m1 + lev * lev * p))

    best = min(uniform_mse(s) for s in np.linspace(0.05, 2.5, 4000))
    assert D <= best + 1e-12


@pytest.mark.parametrize("b", [1, 2, 3, 4, 6, 8])
def test_group_codes_are_nearest_level(b):
    rng = np.random.default_rng(7 + b)
    x = (rng.standard_normal((300, 32)) * np.exp(rng.uniform(-3, 3, (300, 1)))).astype(np.float32)
    codes, scale, zero, bad = lm.quantize_groups(x, b)
    assert not bad.any() and (zero == 0).all()
    L = lm.levels_f16(b).astype(np.float64)
    sf = scale.astype(np.float64)[:, None, None]
    d = np.abs(x.astype(np.float64)[..., None] - L[None, None, :] * sf)
    best = d.min(axis=-1)
    mine = np.take_along_axis(d, codes[..., None].astype(np.int64), axis=-1)[..., 0]
    a = np.abs(x).max(axis=1, keepdims=True).astype(np.float64)
    assert (mine <= best + 2.0 ** -20 * a).all()     # up to the fp32 rounding of a threshold
    # the scale is the group's RMS
    rms = np.sqrt(np.mean(x.astype(np.float64) ** 2, axis=1))
    np.testing.assert_allclose(scale.astype(np.float64), rms, rtol=2.0 ** -10)


def test_group_of_levels_reconstructs_exactly():
    # a group whose values are levels times a power of two, with RMS equal to
    # that power (pairs +-l chosen to give sum l^2 = 32 * 1): exact round trip
    L = lm.levels_f16(1).astype(np.float32)          # +-0.798 (fp16)
    x = np.tile(np.array([L[0], L[1]], np.float32), 16)[None, :] * np.float32(4.0)
    codes, scale, _, _ = lm.quantize_groups(x, 1)
    sf = float(scale[0])
    assert np.array_equal(codes[0], np.tile([0, 1], 16))
    np.testing.assert_array_equal(lm.dequantize_groups(codes, scale, 1)[0],
                                  (L[codes[0]] * np.float32(sf)).astype(np.float32))


def test_zero_and_nonfinite_groups():
    x = np.zeros((2, 32), np.float32)
    x[1, 3] = np.inf
    codes, scale, zero, bad = lm.quantize_groups(x, 3)
    assert (codes == 0).all() and (scale == 0).all() and (zero == 0).all()
    assert list(bad) == [False, True]


def test_lloydmax_mse_fits_the_papers_beta():
    # Sec. 3.1: fitting TurboQuant's Lloyd-Max MSE gives alpha ~ 1.36,
    # beta ~ 3.48 (R^2 > 0.99); the exact D(b), b = 1..6, in ln D = ln alpha - b ln beta
    from oracle import calib
    D = np.array([[lm.design(b)[1] for b in range(1, 9)]])
    a, beta, r2 = calib.fit_distortion(D, 1, 6, 0.0)
    assert beta[0] == pytest.approx(3.48, abs=0.1)
    assert a[0] == pytest.approx(1.36, abs=0.12)
    assert r2[0] > 0.99
