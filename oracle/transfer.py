"""Cross-quantizer transfer matrix (oracle).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Sec. 3.4 "Distortion calibration" (Fig. 3) and App. W "Cross-Quantizer
Transfer" (Table 25): fit (alpha, beta) per quantizer from its own distortion
sweep, allocate with quantizer a's model, and score the bits on quantizer b.
The score is the objective the allocation minimises (Eq. 1) with measured
distortions: J[a][b] = sum_i w_i D_i^b(b_i^a). Composition only: the sweep,
fit and allocation are ``calib`` and ``alloc``.
"""
from __future__ import annotations

import math

import numpy as np

from .alloc import allocate
from .calib import distortion_sweep, fit_distortion
from .quant import ABSMAX, LLOYDMAX, MINMAX, PER_CHANNEL, PER_TOKEN, PER_TOKEN_64, PER_TOKEN_128

# name -> (key grouping, value grouping, hadamard, key form, value form)
FAMILIES = {
    "kivi": (PER_CHANNEL, PER_TOKEN, False, MINMAX, MINMAX),
    "kivi_sym": (PER_CHANNEL, PER_TOKEN, False, ABSMAX, MINMAX),
    "rtn": (PER_TOKEN, PER_TOKEN, False, ABSMAX, ABSMAX),
    "quarot": (PER_TOKEN, PER_TOKEN, True, ABSMAX, ABSMAX),
    "turboquant": (PER_TOKEN, PER_TOKEN, True, LLOYDMAX, LLOYDMAX),
    "turboquant_absmax": (PER_TOKEN_128, PER_TOKEN_64, False, ABSMAX, ABSMAX),
}


def weighted_distortion(w, mse, bits) -> float:
    """sum_i w_i mse[i][b_i - 1], summed in index order in fp64."""
    total = 0.0
    for i, b in enumerate(bits):
        total += float(w[i]) * float(mse[i][int(b) - 1])
    return total


def uniform_bits(n: int, avg_bits: float):
    """Keys (even components) ceil(avg_bits), values floor(avg_bits)."""
    return [math.ceil(avg_bits) if i % 2 == 0 else math.floor(avg_bits) for i in range(n)]


def family_model(x, name, signs, b_lo=2, b_hi=6, r2_min=0.96):
    """mse [n][8], alpha, beta of one family on the sample x [n][T][128]
    (component i is a key when i is even)."""
    kg, vg, had, ks, vs = FAMILIES[name]
    n = x.shape[0]
    mse = distortion_sweep(x, [kg if i % 2 == 0 else vg for i in range(n)], had,
                           signs if had else None,
                           symmetric=[ks if i % 2 == 0 else vs for i in range(n)])
    alpha, beta, _ = fit_distortion(mse, b_lo, b_hi, r2_min, np.arange(n) % 2)
    return mse, alpha, beta


def transfer_matrix(x, w, avg_bits, allowed_mask, signs=None, names=None, b_lo=2, b_hi=6,
                    r2_min=0.96):
    names = list(names or FAMILIES)
    res = {"names": names, "mse": {}, "alpha": {}, "beta": {}, "bits": {}}
    for f in names:
        mse, alpha, beta = family_model(x, f, signs, b_lo, b_hi, r2_min)
        bits, _ = allocate(w, alpha, beta, avg_bits, allowed_mask)
        res["mse"][f], res["alpha"][f], res["beta"][f], res["bits"][f] = mse, alpha, beta, bits
    res["J"] = {a: {b: weighted_distortion(w, res["mse"][b], res["bits"][a]) for b in names}
                for a in names}
    ub = uniform_bits(x.shape[0], avg_bits)
    res["uniform"] = {b: weighted_distortion(w, res["mse"][b], ub) for b in names}
    return res
