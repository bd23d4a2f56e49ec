"""Pins for the cross-quantizer transfer matrix (CPU only).

The matched allocation minimises its own fitted objective over every integer
allocation of the budget (Prop. 3: greedy is optimal for convex separable
costs), checked by brute force on a handful of components; the allocation is
invariant to a common scale of the distortions (only beta and ratios of
w alpha matter); every allocation spends exactly the budget; and on the
synthetic cache, whose quantizers have different betas (Sec. 3.4), a
mismatched model moves bits and costs distortion.
"""
import itertools
import math

import numpy as np
import pytest

from oracle import alloc as oalloc
from oracle import transfer as otr
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.workloads import LLAMA3_8B_32K

ALLOWED = (2, 3, 4)
MASK = sum(1 << b for b in ALLOWED)


@pytest.fixture(scope="module")
def sample():
    wl = LLAMA3_8B_32K.scaled(L=1, H_kv=3)
    x = synth.calibration_sample(wl, T=64).float().numpy()      # 6 components
    w = synth.importances(x.shape[0], 0.74, 5)
    signs = synth.hadamard_signs(5).numpy()
    return x, w, signs


@pytest.fixture(scope="module")
def matrix(sample):
    x, w, signs = sample
    return otr.transfer_matrix(x, w, 3.0, MASK, signs)


def model_cost(w, alpha, beta, bits):
    return sum(w[i] * alpha[i] * beta[i] ** (-int(b)) for i, b in enumerate(bits))


def test_matched_allocation_is_the_brute_force_optimum(sample, matrix):
    x, w, _ = sample
    n = x.shape[0]
    B = oalloc.budget(3.0, n)
    for f in matrix["names"]:
        a, b = matrix["alpha"][f], matrix["beta"][f]
        best = min(model_cost(w, a, b, c) for c in itertools.product(ALLOWED, repeat=n)
                   if sum(c) == B)
        got = model_cost(w, a, b, matrix["bits"][f])
        assert got == pytest.approx(best, rel=1e-12), f
        for g in matrix["names"]:                      # no other family's bits do better
            assert got <= model_cost(w, a, b, matrix["bits"][g]) * (1 + 1e-12)


def test_every_allocation_spends_the_budget(sample, matrix):
    n = sample[0].shape[0]
    for f in matrix["names"]:
        assert sum(int(b) for b in matrix["bits"][f]) == oalloc.budget(3.0, n)
        assert set(int(b) for b in matrix["bits"][f]) <= set(ALLOWED)
    assert sum(otr.uniform_bits(n, 2.5)) == oalloc.budget(2.5, n)


def test_common_scale_leaves_allocation_unchanged(sample):
    x, w, signs = sample
    mse, alpha, beta = otr.family_model(x, "rtn", signs)
    from oracle.calib import fit_distortion
    a2, b2, _ = fit_distortion(mse * 7.0, 2, 6, 0.96, np.arange(x.shape[0]) % 2)
    np.testing.assert_allclose(b2, beta, rtol=1e-12)
    np.testing.assert_allclose(a2, 7.0 * alpha, rtol=1e-12)
    b1, _ = oalloc.allocate(w, alpha, beta, 3.0, MASK)
    b7, _ = oalloc.allocate(w, a2, b2, 3.0, MASK)
    assert list(b1) == list(b7)


def test_weighted_distortion_by_hand():
    w = [1.0, 2.0]
    mse = [[8.0, 4.0, 2.0, 1.0, 0, 0, 0, 0], [9.0, 3.0, 1.0, 0.5, 0, 0, 0, 0]]
    assert otr.weighted_distortion(w, mse, [2, 3]) == 4.0 + 2.0 * 1.0
    assert otr.uniform_bits(4, 2.5) == [3, 2, 3, 2]
    assert otr.uniform_bits(3, 3.0) == [3, 3, 3]


def test_mismatched_beta_moves_bits_and_costs_distortion(sample, matrix):
    # the synthetic cache gives per-token keys a much smaller beta than
    # per-channel keys (outlier channels), as TurboQuant's 3.6 vs KIVI's 5.1
    bk = {f: float(np.mean(matrix["beta"][f][0::2])) for f in matrix["names"]}
    assert bk["rtn"] < 4.0 < bk["kivi"]
    J = matrix["J"]
    moved = [(a, b) for a in matrix["names"] for b in matrix["names"]
             if list(matrix["bits"][a]) != list(matrix["bits"][b])]
    assert moved
    # scored on the quantizer that holds the bits, some foreign model loses
    # more than 5 % against the matched one
    worse = [J[a][b] / J[b][b] for a, b in moved]
    assert max(worse) > 1.05
