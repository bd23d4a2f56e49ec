"""Lloyd-Max scalar codebook quantizer (oracle).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Paper passages followed
-----------------------
* App. F Table 8: the exact Lloyd-Max MSE of a unit-variance Gaussian source
  at b = 1..6 bits; Sec. 3.1 (after Assumption 1) fits it with
  alpha ~ 1.36, beta ~ 3.48.
* Sec. 2 / Sec. 4.1 and App. W: TurboQuant rotates and then applies a
  Lloyd-Max scalar quantizer per coordinate ("per-token ... Lloyd-Max").

Codebook: the 2^b-level Lloyd-Max quantizer of N(0, 1) (Lloyd's method /
Max 1960): levels l_0 < ... < l_{n-1} that satisfy both optimality
conditions,
    t_i = (l_{i-1} + l_i) / 2                   (nearest-level cells)
    l_i = E[X | t_i <= X < t_{i+1}]
        = (phi(t_i) - phi(t_{i+1})) / (Phi(t_{i+1}) - Phi(t_i))   (centroids)
with t_0 = -inf, t_n = +inf; found by Lloyd's iteration from the quantile
initialisation l_i = Phi^-1((i + 1/2) / n) and then Newton's method on the
same fixed point, in fp64. Its MSE is D(b) = 1 - sum_i p_i l_i^2 (the
centroid condition makes the cross terms vanish).

Group quantizer (the reading used here; the paper gives no per-group
normalisation for this quantizer, and TurboQuant scales by the vector
norm): for one group x[0..31], with v = fp32(x) + 0 as in ``quant``,
    s2    = fp32(S(0..15) + S(16..31)), S(i..j) = the fp32 sum of fp32(v_k * v_k)
            for k = i..j in this order (two halves, added last)
    scale = fp16(fp32_sqrt(s2 / 32)),  zero = +0         (the group's RMS)
    L_c   = fp16(l_c)                                     (stored levels)
    T_i   = fp32(fp32((L_{i-1} + L_i) / 2) * sf),  i = 1..n-1
    code  = #{i : v >= T_i}      (a value on a threshold takes the upper level)
    x_hat = fp32(L_code * sf) + 0
A group of zeros (sf == 0) gets codes 0; a non-finite value or an fp16
overflow of the scale is a numeric failure (codes 0, scale 0, zero 0).
"""
from __future__ import annotations

import math

import numpy as np
from scipy.special import ndtr, ndtri

GROUP = 32


def _phi(t):
    return np.exp(-0.5 * t * t) / math.sqrt(2.0 * math.pi)


def _centroids(lev):
    """Thresholds t, cell probabilities p and centroids C(lev) of N(0, 1).
    Cells above 0 take their probability from the upper tail, Phi(-t_i) -
    Phi(-t_{i+1}), which keeps its digits far out."""
    t = np.concatenate([[-np.inf], 0.5 * (lev[:-1] + lev[1:]), [np.inf]])
    lo, hi = t[:-1], t[1:]
    upper = lo >= 0
    p = np.where(upper, ndtr(-lo) - ndtr(-hi), ndtr(hi) - ndtr(lo))
    return t, p, (_phi(lo) - _phi(hi)) / p


def design(b: int, lloyd_steps: int = 200, newton_steps: int = 50):
    """Lloyd-Max levels of N(0, 1) at b bits (fp64, ascending) and their MSE.

    Lloyd's iteration lev <- C(lev) from the quantile start, then Newton's
    method on the same fixed point, F(lev) = lev - C(lev) = 0, whose Jacobian
    is tridiagonal (C_i depends on the thresholds t_i, t_{i+1}, i.e. on
    lev_{i-1}, lev_i, lev_{i+1}): dC_i/dt_i = phi(t_i) (C_i - t_i) / p_i,
    dC_i/dt_{i+1} = phi(t_{i+1}) (t_{i+1} - C_i) / p_i, each threshold half of
    its two levels. Plain Lloyd converges too slowly at 7-8 bits.
    """
    n = 2 ** b
    lev = ndtri((np.arange(n) + 0.5) / n)
    for _ in range(lloyd_steps):
        lev = _centroids(lev)[2]
    for _ in range(newton_steps):
        t, p, c = _centroids(lev)
        F = lev - c
        ta = np.where(np.isfinite(t[:-1]), t[:-1], 0.0)      # the infinite ends add nothing
        tc = np.where(np.isfinite(t[1:]), t[1:], 0.0)
        ga = np.where(np.isfinite(t[:-1]), _phi(ta) * (c - ta) / p, 0.0)    # dC_i/dt_i
        gc = np.where(np.isfinite(t[1:]), _phi(tc) * (tc - c) / p, 0.0)     # dC_i/dt_{i+1}
        lower = -0.5 * ga[1:]                 # J[i][i-1], i = 1..n-1
        diag = 1.0 - 0.5 * (ga + gc)
        upper = -0.5 * gc[:-1]                # J[i][i+1], i = 0..n-2
        step = _solve_tridiagonal(lower, diag, upper, -F)
        lev = lev + step
        if np.max(np.abs(step)) < 1e-15:
            break
    lev = 0.5 * (lev - lev[::-1])          # the source is symmetric, so is the codebook
    t, p, c = _centroids(lev)
    return lev, float(1.0 - np.sum(p * lev * lev))


def _solve_tridiagonal(lower, diag, upper, rhs):
    """Thomas algorithm for a tridiagonal system (fp64)."""
    n = diag.size
    cp = np.zeros(n)
    dp = np.zeros(n)
    cp[0] = upper[0] / diag[0] if n > 1 else 0.0
    dp[0] = rhs[0] / diag[0]
    for i in range(1, n):
        m = diag[i] - lower[i - 1] * cp[i - 1]
        cp[i] = upper[i] / m if i < n - 1 else 0.0
        dp[i] = (rhs[i] - lower[i - 1] * dp[i - 1]) / m
    x = np.zeros(n)
    x[-1] = dp[-1]
    for i in range(n - 2, -1, -1):
        x[i] = dp[i] - cp[i] * x[i + 1]
    return x


_CODEBOOKS: dict[int, np.ndarray] = {}


def levels_f16(b: int) -> np.ndarray:
    """The stored codebook: fp16 levels L_0 < ... < L_{2^b - 1}."""
    if b not in _CODEBOOKS:
        _CODEBOOKS[b] = design(b)[0].astype(np.float16)
    return _CODEBOOKS[b]


def quantize_groups(v: np.ndarray, b: int):
    """Groups along the last axis (length 32). Returns (codes uint8, scale
    float16, zero float16, bad bool) like ``quant.quantize_groups``."""
    assert 1 <= b <= 8
    v = (np.asarray(v, dtype=np.float32) + np.float32(0.0)).astype(np.float32)
    assert v.shape[-1] == GROUP
    L = levels_f16(b).astype(np.float32)
    with np.errstate(all="ignore"):
        finite = np.isfinite(v).all(axis=-1)
        vv = np.where(finite[..., None], v, np.float32(0.0))
        halves = []
        for h in range(2):                           # each half summed in order, in fp32
            acc = np.zeros(vv.shape[:-1], dtype=np.float32)
            for i in range(16 * h, 16 * h + 16):
                acc = (acc + (vv[..., i] * vv[..., i]).astype(np.float32)).astype(np.float32)
            halves.append(acc)
        s2 = (halves[0] + halves[1]).astype(np.float32)
        rms = np.sqrt((s2 / np.float32(GROUP)).astype(np.float32)).astype(np.float32)
        scale = rms.astype(np.float16)
        bad = (~finite) | (~np.isfinite(scale))
        sf = np.where(bad, np.float32(0.0), scale.astype(np.float32)).astype(np.float32)
        mids = ((L[:-1] + L[1:]) / np.float32(2.0)).astype(np.float32)           # exact
        T = (mids[None, :] * sf.reshape(-1, 1)).astype(np.float32)               # [groups][n-1]
        flat = vv.reshape(-1, GROUP)
        codes = (flat[:, :, None] >= T[:, None, :]).sum(axis=-1)
        ok = (~bad.reshape(-1)) & (sf.reshape(-1) != 0)
        codes = np.where(ok[:, None], codes, 0).reshape(vv.shape).astype(np.uint8)
    scale = np.where(bad, np.float16(0.0), scale).astype(np.float16)
    zero = np.zeros_like(scale, dtype=np.float16)
    return codes, scale, zero, bad


def dequantize_groups(codes: np.ndarray, scale: np.ndarray, b: int) -> np.ndarray:
    """x_hat = fp32(L_code * sf) (+ zero, which is +0)."""
    L = levels_f16(b).astype(np.float32)
    sf = np.asarray(scale, dtype=np.float16).astype(np.float32)[..., None]
    return (L[codes.astype(np.int64)] * sf).astype(np.float32)
