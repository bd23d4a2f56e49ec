"""Pins for the oracle's distortion sweep and log-linear fit (CPU only)."""
import math
import os

import numpy as np
import pytest

from oracle import calib
from oracle.quant import PER_CHANNEL, PER_TOKEN

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _table8():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "table8_lloydmax.txt"))
            if l.strip() and not l.startswith("#")]
    b = np.array([int(r[0]) for r in rows])
    exact = np.array([float(r[1]) for r in rows])
    fit = np.array([float(r[2]) for r in rows])
    ratio = np.array([float(r[3]) for r in rows])
    return b, exact, fit, ratio


def test_table8_fit_reproduces_paper():
    # Sec. 3.1 / App. F Table 8: fitting the exact Lloyd-Max D(b), b = 1..6,
    # gives alpha ~ 1.36, beta ~ 3.48, R^2 > 0.99, and the "Fit" column.
    b, exact, fit, ratio = _table8()
    row = np.zeros(8)
    row[:6] = exact
    a, beta, r2 = calib.fit_one(row, 1, 6)
    assert abs(a - 1.36) < 0.005
    assert abs(beta - 3.48) < 0.005
    assert r2 > 0.99
    model = a * beta ** (-b.astype(float))
    assert np.all(np.abs(model / fit - 1.0) < 3e-3)      # printed to 4 digits
    assert np.all(np.abs(model / exact - ratio) < 5e-3)     # Ratio = Fit / Exact
    # 1/ln(beta) ~ 0.80 extra bits per e-fold of sensitivity (Sec. 3.1).
    assert abs(1.0 / math.log(beta) - 0.80) < 0.005


def test_exact_exponential_recovered():
    row = [2.5 * 4.2 ** (-k) for k in range(1, 9)]
    for lo, hi in ((2, 6), (1, 8), (3, 4)):
        a, beta, r2 = calib.fit_one(row, lo, hi)
        assert abs(a / 2.5 - 1) < 1e-12 and abs(beta / 4.2 - 1) < 1e-12
        assert abs(r2 - 1.0) < 1e-12


def test_degenerate_rows():
    a, beta, r2 = calib.fit_one([0.0] * 8, 2, 6)
    assert a == 0.0 and beta == math.inf and r2 == 1.0
    row = [0.1, 0.02, 0, 0, 0, 0, 0, 0]
    a, beta, r2 = calib.fit_one(row, 2, 6)          # one positive point only
    assert beta == math.inf
    row = [0.5] * 8                                  # flat: beta = 1, R^2 = 1
    a, beta, r2 = calib.fit_one(row, 2, 6)
    assert abs(beta - 1.0) < 1e-15 and r2 == 1.0


def test_poor_fit_fallback_per_class():
    # App. W "Outlier heads": R^2 < 0.96 -> beta = min(beta_fit, beta_bar),
    # beta_bar = mean fitted beta of the component's class.
    good_k = [3.0 * 5.0 ** (-k) for k in range(1, 9)]
    good_v = [3.0 * 4.0 ** (-k) for k in range(1, 9)]
    bad = [1.0, 0.9, 1e-3, 1e-2, 1e-6, 1e-5, 1e-9, 1e-9]   # zig-zag
    mse = np.array([good_k, good_v, bad, bad])
    classes = [0, 1, 0, 1]
    a, beta, r2 = calib.fit_distortion(mse, 2, 6, 0.96, classes)
    a0, b_bad, r2_bad = calib.fit_one(bad, 2, 6)
    assert r2_bad < 0.96 and b_bad > 5.0
    assert abs(beta[0] - 5.0) < 1e-12 and abs(beta[1] - 4.0) < 1e-12
    assert abs(beta[2] - min(b_bad, (5.0 + b_bad) / 2)) < 1e-12
    assert abs(beta[3] - min(b_bad, (4.0 + b_bad) / 2)) < 1e-12
    # r2_min <= 0 disables the fallback
    a, beta2, _ = calib.fit_distortion(mse, 2, 6, 0.0, classes)
    assert abs(beta2[2] - b_bad) < 1e-12


def test_sweep_constant_and_uniform():
    # Constant components have zero distortion at every b. Uniform data where
    # every group of 32 spans exactly [0, 1] (one 0 and one 1 per group):
    # the other 30 elements have error uniform on [-s/2, s/2], so
    # D(b) = (30/32) s^2 / 12 (3-sigma of the estimate ~ 1.5%).
    x = np.zeros((2, 512, 128), dtype=np.float32)
    x[0] = 0.75
    rng = np.random.default_rng(2)
    u = rng.random((512, 128)).astype(np.float32)
    u[:, 0::32] = 0.0
    u[:, 1::32] = 1.0
    x[1] = u
    mse = calib.distortion_sweep(x, [PER_TOKEN, PER_TOKEN])
    assert (mse[0] == 0).all()
    for b in (3, 4, 6):
        s = float(np.float16(np.float32(1.0) / np.float32(2 ** b - 1)))
        assert abs(mse[1, b - 1] / (30.0 / 32.0 * s * s / 12) - 1) < 0.02


def test_sweep_monotone_and_beta_range():
    rng = np.random.default_rng(8)
    x = rng.standard_normal((2, 512, 128)).astype(np.float32)
    mse = calib.distortion_sweep(x, [PER_CHANNEL, PER_TOKEN])
    assert np.all(np.diff(mse, axis=1) < 0)
    a, beta, r2 = calib.fit_distortion(mse, 2, 6, 0.96)
    # high-rate uniform quantization: step halves per bit -> D ratio -> 4
    assert np.all(beta > 3.9) and np.all(beta < 4.6)
    assert np.all(r2 > 0.99)
