"""Pins for the oracle's allocators (CPU only): brute force, closed forms,
the paper's printed numbers."""
import itertools
import math

import numpy as np
import pytest

from oracle import alloc


def _brute(w, a, beta, B, allowed):
    best = math.inf
    arg = None
    for bits in itertools.product(allowed, repeat=len(w)):
        if sum(bits) != B:
            continue
        J = alloc.objective(w, a, beta, bits)
        if J < best:
            best, arg = J, bits
    return best, arg


def _instance(rng, n):
    w = np.exp(rng.normal(0, 0.8, n))
    a = rng.uniform(0.5, 20.0, n)
    beta = rng.uniform(3.0, 6.0, n)
    return list(w), list(a), list(beta)


@pytest.mark.parametrize("seed", range(12))
def test_greedy_equals_brute_force(seed):
    # Prop. 3: greedy is optimal for convex D (contiguous bit set).
    rng = np.random.default_rng(seed)
    n = int(rng.integers(2, 7))
    w, a, beta = _instance(rng, n)
    allowed = [2, 3, 4]
    for B in range(2 * n, 4 * n + 1):
        bits = alloc.greedy(w, a, beta, B, 2, 4)
        J = alloc.objective(w, a, beta, bits)
        best, _ = _brute(w, a, beta, B, allowed)
        assert sum(bits) == B and min(bits) >= 2 and max(bits) <= 4
        assert abs(J - best) <= 1e-12 * best


@pytest.mark.parametrize("seed", range(12))
def test_dp_equals_brute_force_noncontiguous(seed):
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(2, 7))
    w, a, beta = _instance(rng, n)
    allowed = [2, 3, 4, 8]
    for B in range(2 * n, 8 * n + 1):
        best, _ = _brute(w, a, beta, B, allowed)
        bits = alloc.dp(w, a, beta, B, allowed)
        if best == math.inf:
            assert bits is None
            continue
        assert sum(bits) == B and set(bits) <= set(allowed)
        assert abs(alloc.objective(w, a, beta, bits) - best) <= 1e-12 * best


def test_dp_matches_greedy_on_contiguous_sets():
    rng = np.random.default_rng(5)
    w, a, beta = _instance(rng, 40)
    for B in (80, 95, 120, 150, 160):
        g = alloc.greedy(w, a, beta, B, 2, 4)
        d = alloc.dp(w, a, beta, B, [2, 3, 4])
        assert abs(alloc.objective(w, a, beta, g) - alloc.objective(w, a, beta, d)) <= \
            1e-12 * alloc.objective(w, a, beta, g)


def test_equal_components_spread_lowest_index_first():
    n = 10
    bits = alloc.greedy([1.0] * n, [1.0] * n, [4.0] * n, 34, 2, 6)
    assert bits == [4, 4, 4, 4, 3, 3, 3, 3, 3, 3]
    bits = alloc.dp([1.0] * n, [1.0] * n, [4.0] * n, 34, [2, 3, 4, 5, 6])
    assert bits == [4, 4, 4, 4, 3, 3, 3, 3, 3, 3]


def test_budget_and_R_of_the_paper():
    # Sec. 3.3: Qwen3-8B, N = 288 heads (576 K/V components), b_bar = 4,
    # b_min = 2 -> R = 2N(b_bar - b_min) = 1152 greedy steps.
    n = 576
    assert alloc.budget(4.0, n) - n * 2 == 1152
    rng = np.random.default_rng(0)
    w, a, beta = _instance(rng, n)
    bits = alloc.greedy(w, a, beta, alloc.budget(4.0, n), 2, 6)
    assert sum(bits) == 2304 and sum(b - 2 for b in bits) == 1152
    # B = round(b_bar * n): 2.5 * 512 = 1280, 3.0 * 1280 = 3840
    assert alloc.budget(2.5, 512) == 1280 and alloc.budget(3.0, 1280) == 3840
    assert alloc.budget(2.5, 5) == 13          # 12.5 rounds half up


def test_infeasible_budgets():
    w, a, beta = [1.0] * 3, [1.0] * 3, [4.0] * 3
    assert alloc.greedy(w, a, beta, 5, 2, 4) is None
    assert alloc.greedy(w, a, beta, 13, 2, 4) is None
    assert alloc.dp(w, a, beta, 5, [2, 8]) is None
    assert alloc.dp(w, a, beta, 7, [2, 8]) is None      # 6 + {0, 6, 12, 18}
    assert alloc.dp(w, a, beta, 12, [2, 8]) == [8, 2, 2]


def test_continuous_equation_2():
    # Thm. 1 Eq. 2: shared beta and inactive bounds ->
    # b_i = b_bar + (ln w_i - mean ln w) / ln beta.
    rng = np.random.default_rng(3)
    n = 64
    w = np.exp(rng.normal(0, 0.5, n))
    beta = 4.7
    out = alloc.continuous(list(w), [2.0] * n, [beta] * n, 4.0, 0.0, 8.0)
    lw = np.log(w)
    ref = 4.0 + (lw - lw.mean()) / math.log(beta)
    assert np.allclose(out, ref, rtol=0, atol=1e-12)
    assert abs(sum(out) - 4.0 * n) < 1e-9


def test_continuous_printed_shifts():
    # Sec. 3.1: an e-fold more sensitive head gets 1/ln 3.48 ~ 0.80 more bits;
    # Sec. 3.4: a 2x sensitivity error shifts by ln 2 / ln 5 ~ 0.43 bits.
    out = alloc.continuous([1.0, math.e], [1.0, 1.0], [3.48, 3.48], 4.0, 0.0, 8.0)
    assert abs((out[1] - out[0]) - 0.80) < 0.005
    out = alloc.continuous([1.0, 2.0], [1.0, 1.0], [5.0, 5.0], 4.0, 0.0, 8.0)
    assert abs((out[1] - out[0]) - 0.43) < 0.005


def test_continuous_kkt_with_bounds():
    # App. B.1 iterative clipping: free components share the multiplier
    # lambda = w alpha ln(beta) beta^-b; clipped ones sit on a bound and
    # would move past it; the budget holds.
    rng = np.random.default_rng(4)
    n = 50
    w = list(np.exp(rng.normal(0, 1.5, n)))
    a = list(rng.uniform(1, 10, n))
    beta = list(rng.uniform(3.5, 5.5, n))
    out = alloc.continuous(w, a, beta, 3.0, 2.0, 4.0)
    assert abs(sum(out) - 150.0) < 1e-9
    lam = [w[i] * a[i] * math.log(beta[i]) * beta[i] ** (-out[i]) for i in range(n)]
    free = [i for i in range(n) if 2.0 < out[i] < 4.0]
    assert len(free) > 5
    lf = [lam[i] for i in free]
    assert max(lf) / min(lf) - 1 < 1e-9
    for i in range(n):
        if out[i] == 2.0:
            assert lam[i] <= lf[0] * (1 + 1e-9)
        if out[i] == 4.0:
            assert lam[i] >= lf[0] * (1 - 1e-9)


def test_gain_ratio_amgm():
    # Thm. 2: J_uniform / J_opt = AM(w) / GM(w) (continuous, no active bounds).
    rng = np.random.default_rng(6)
    n = 200
    w = list(np.exp(rng.normal(0, 0.7, n)))
    beta = 5.1
    opt = alloc.continuous(w, [1.0] * n, [beta] * n, 4.0, -100.0, 100.0)
    Ju = sum(x * beta ** -4.0 for x in w)             # every b_i = b_bar = 4
    Jopt = sum(w[i] * beta ** (-opt[i]) for i in range(n))
    assert abs((Ju / Jopt) / alloc.am_gm(w) - 1) < 1e-10


def test_lognormal_gain_corollary():
    # Cor. 1: ln w ~ N(mu, sigma^2) -> AM/GM -> exp(sigma^2 / 2);
    # sigma = 0.76 (Qwen3-8B, App. R) -> 1.335.
    rng = np.random.default_rng(7)
    w = np.exp(rng.normal(0.3, 0.76, 400000))
    assert abs(alloc.am_gm(list(w)) / math.exp(0.76 ** 2 / 2) - 1) < 0.01
    assert abs(math.exp(0.76 ** 2 / 2) - 1.335) < 0.001


def test_cap_and_allocate_dispatch():
    # App. W "Mitigation": w_i <- min(w_i, 5 w_bar).
    w = [1.0] * 9 + [100.0]
    capped = alloc.cap_weights(w)
    assert capped[:9] == [1.0] * 9 and capped[9] == 5.0 * 109.0 / 10.0
    mask = (1 << 2) | (1 << 3) | (1 << 4)
    n = len(w)
    bits, J = alloc.allocate(w, [1.0] * n, [4.0] * n, 3.0, mask)
    assert sum(bits) == 30 and bits[9] == 4
    mask8 = mask | (1 << 8)
    bits8, _ = alloc.allocate(w, [1.0] * n, [4.0] * n, 3.5, mask8)
    assert sum(bits8) == 35 and set(bits8) <= {2, 3, 4, 8}
    assert alloc.allocate(w, [1.0] * n, [4.0] * n, 9.0, mask)[0] is None
    bc, _ = alloc.allocate(w, [1.0] * n, [4.0] * n, 3.0, mask, cap=True)
    assert sum(bc) == 30
