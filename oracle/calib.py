"""Distortion calibration (oracle): MSE sweep D_i(b) and fit of D(b) = alpha beta^-b.

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Paper passages followed
-----------------------
* Assumption 1: the per-head quantization MSE follows D(b) = alpha * beta^-b
  with alpha > 0, beta > 1.
* Alg. 1 stage 2 and Sec. 3.4 "Distortion calibration": measure the MSE at
  b in {2,...,6} and fit by least squares on ln D = ln alpha - b ln beta.
* App. W "Outlier heads": heads with R^2 < 0.96 use beta = min(beta_fit, beta_bar).
* App. F Table 8 (Lloyd-Max, d = 128): the exact D(b) column is the pin for
  the fit; the paper reports alpha ~ 1.36, beta ~ 3.48.

Readings where the paper is silent
----------------------------------
* D_i(b) is the per-element MSE over all elements of component i, measured in
  the quantizer's own domain (after rotation when rotating):
  D = sum((fp64(y) - fp64(x_hat))^2) / (T * 128).
* The fit uses unweighted least squares over the b in [b_lo, b_hi] whose
  D(b) > 0. With fewer than two such points: alpha = 0, beta = +inf, R^2 = 1
  (zero distortion model).
* R^2 = 1 - SS_res / SS_tot on ln D; SS_tot = 0 gives R^2 = 1.
* beta_bar is the arithmetic mean of the fitted (finite) beta over the
  components of the same class (K or V), taken before any fallback.
"""
from __future__ import annotations

import math

import numpy as np

from .quant import quantize_stream


def distortion_sweep(x: np.ndarray, groupings, hadamard: bool = False, signs=None,
                     bits=range(1, 9), symmetric=False) -> np.ndarray:
    """x [n][T][128] (fp16/bf16 values as fp32); groupings[n] in {PER_TOKEN, PER_CHANNEL};
    ``symmetric``: the quantizer form (``quant.MINMAX`` / ``ABSMAX`` /
    ``LLOYDMAX``; a bool means min-max / absmax), one, or one per component.

    Returns mse [n][len(bits)] float64.
    """
    x = np.asarray(x, dtype=np.float32)
    n = x.shape[0]
    bits = list(bits)
    sym = np.broadcast_to(np.asarray(symmetric, dtype=np.int64), (n,))
    out = np.zeros((n, len(bits)), dtype=np.float64)
    for i in range(n):
        for k, b in enumerate(bits):
            r = quantize_stream(x[i], int(groupings[i]), b, signs, hadamard, int(sym[i]))
            err = r["y"].astype(np.float64) - r["xhat"].astype(np.float64)
            out[i, k] = float(np.sum(err * err)) / err.size
    return out


def fit_one(mse_row, b_lo: int, b_hi: int):
    """Least-squares fit of ln D on b for one component (plain loops, fp64).

    ``mse_row[k]`` is D(k+1). Returns (alpha, beta, r2).
    """
    pts = [(float(b), math.log(float(mse_row[b - 1])))
           for b in range(b_lo, b_hi + 1) if float(mse_row[b - 1]) > 0.0]
    n = len(pts)
    if n < 2:
        return 0.0, math.inf, 1.0
    sb = 0.0
    sy = 0.0
    for b, y in pts:
        sb += b
        sy += y
    mb = sb / n
    my = sy / n
    sxy = 0.0
    sxx = 0.0
    for b, y in pts:
        sxy += (b - mb) * (y - my)
        sxx += (b - mb) * (b - mb)
    m = sxy / sxx
    c = my - m * mb
    ss_res = 0.0
    ss_tot = 0.0
    for b, y in pts:
        r = y - (c + m * b)
        ss_res += r * r
        ss_tot += (y - my) * (y - my)
    if ss_tot == 0.0:
        r2 = 1.0 if ss_res == 0.0 else 0.0
    else:
        r2 = 1.0 - ss_res / ss_tot
    return math.exp(c), math.exp(-m), r2


def fit_distortion(mse: np.ndarray, b_lo: int = 2, b_hi: int = 6, r2_min: float = 0.96,
                   classes=None):
    """Fit every component; apply the poor-fit fallback per class.

    ``mse`` [n][8] with column k = D(k+1). ``classes`` [n] ints (None: one class).
    Returns (alpha[n], beta[n], r2[n]) float64.
    """
    mse = np.asarray(mse, dtype=np.float64)
    n = mse.shape[0]
    alpha = np.zeros(n)
    beta = np.zeros(n)
    r2 = np.zeros(n)
    for i in range(n):
        alpha[i], beta[i], r2[i] = fit_one(mse[i], b_lo, b_hi)
    if classes is None:
        classes = [0] * n
    if r2_min > 0.0:
        means = {}
        for cl in sorted(set(int(c) for c in classes)):
            s = 0.0
            k = 0
            for i in range(n):
                if int(classes[i]) == cl and math.isfinite(beta[i]):
                    s += beta[i]
                    k += 1
            means[cl] = s / k if k > 0 else math.inf
        fitted = beta.copy()
        for i in range(n):
            if r2[i] < r2_min:
                beta[i] = min(fitted[i], means[int(classes[i])])
    return alpha, beta, r2
