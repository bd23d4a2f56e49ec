"""Bit allocation (oracle): reverse waterfilling, integer greedy, exact DP.

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Paper passages followed
-----------------------
* Eq. 1: minimise J(b) = sum_i w_i D_i(b_i) s.t. sum_i b_i = B,
  b_min <= b_i <= b_max, with B = round(b_bar * N).
* Thm. 1, Eq. 2 and App. B.1: continuous optimum
  b_i = (ln(w_i alpha_i ln beta_i) - ln lambda) / ln beta_i; with one shared beta
  this is b_i = b_bar + (ln w_i - mean ln w) / ln beta. Bounds: iterative
  clip-and-redistribute (App. B.1 "Iterative waterfilling", Sec. 3.4).
* Alg. 1 stage 3, Sec. 3.3, Alg. 2: greedy integer allocation; start at b_min,
  repeatedly give one bit to the component with the largest marginal gain
  w_i alpha_i beta_i^-b_i (1 - beta_i^-1), max-heap, R = B - 2N b_min steps.
* Prop. 3 / App. B.3: greedy is optimal when D is convex (used as a check).
* Sec. 3.4 "K/V separation": keys and values are separate components sharing
  one budget (the component index already encodes this).
* App. W "Mitigation": optional cap w_i <- min(w_i, 5 w_bar).
* Thm. 2 / Cor. 1: J_uniform / J_opt = AM(w) / GM(w); exp(sigma^2 / 2) for
  log-normal w.

Readings where the paper is silent
----------------------------------
* B = floor(b_bar * n + 0.5) (the paper writes the rounding bracket).
* Greedy ties: equal gains go to the lower component index.
* A non-contiguous allowed set (e.g. {2,3,4,8}) cannot be walked one bit at a
  time; the exact optimum is found by a dynamic programme over components
  and spent budget. Ties: the larger bit-width for the lower index (the same
  preference as the greedy's tie rule). Floating-point comparisons are exact
  on values computed in a fixed order (cost first, then one addition).
"""
from __future__ import annotations

import heapq
import math

import numpy as np


def budget(avg_bits: float, n: int) -> int:
    return int(math.floor(avg_bits * n + 0.5))


def allowed_bits(mask: int):
    return [k for k in range(1, 9) if (mask >> k) & 1]


def is_contiguous(bits) -> bool:
    return len(bits) > 0 and bits == list(range(bits[0], bits[-1] + 1))


def cap_weights(w):
    w = [float(x) for x in w]
    mean = 0.0
    for x in w:
        mean += x
    mean /= len(w)
    return [min(x, 5.0 * mean) for x in w]


def gain(w: float, a: float, beta: float, b: int) -> float:
    """Marginal gain of the (b+1)-th bit: w alpha beta^-b (1 - 1/beta)."""
    return ((w * a) * math.pow(beta, -float(b))) * (1.0 - 1.0 / beta)


def cost(w: float, a: float, beta: float, b: int) -> float:
    """w alpha beta^-b."""
    return (w * a) * math.pow(beta, -float(b))


def objective(w, alpha, beta, bits) -> float:
    s = 0.0
    for i in range(len(bits)):
        s += cost(float(w[i]), float(alpha[i]), float(beta[i]), int(bits[i]))
    return s


def greedy(w, alpha, beta, B: int, b_min: int, b_max: int):
    """Alg. 2: max-heap greedy. Returns list of ints, or None if infeasible."""
    n = len(w)
    if B < n * b_min or B > n * b_max:
        return None
    bits = [b_min] * n
    R = B - n * b_min
    heap = []
    if b_min < b_max:
        for i in range(n):
            heapq.heappush(heap, (-gain(w[i], alpha[i], beta[i], b_min), i))
    while R > 0:
        _, i = heapq.heappop(heap)
        bits[i] += 1
        R -= 1
        if bits[i] < b_max:
            heapq.heappush(heap, (-gain(w[i], alpha[i], beta[i], bits[i]), i))
    return bits


def dp(w, alpha, beta, B: int, allowed):
    """Exact integer optimum over an arbitrary allowed set (suffix DP).

    g[i][r] = least cost of components i..n-1 with r extra bits above min.
    Returns list of ints, or None if B is unreachable.
    """
    n = len(w)
    allowed = sorted(allowed)
    lo = allowed[0]
    R = B - n * lo
    if R < 0:
        return None
    inf = math.inf
    g = [[inf] * (R + 1) for _ in range(n + 1)]
    g[n][0] = 0.0
    costs = [[cost(w[i], alpha[i], beta[i], s) for s in allowed] for i in range(n)]
    for i in range(n - 1, -1, -1):
        gi = g[i]
        gn = g[i + 1]
        ci = costs[i]
        for r in range(R + 1):
            best = inf
            for k, s in enumerate(allowed):
                d = s - lo
                if d > r or gn[r - d] == inf:
                    continue
                v = ci[k] + gn[r - d]
                if v < best:
                    best = v
            gi[r] = best
    if g[0][R] == inf:
        return None
    bits = []
    r = R
    for i in range(n):
        for k in range(len(allowed) - 1, -1, -1):
            s = allowed[k]
            d = s - lo
            if d > r or g[i + 1][r - d] == inf:
                continue
            if costs[i][k] + g[i + 1][r - d] == g[i][r]:
                bits.append(s)
                r -= d
                break
    return bits


def allocate(w, alpha, beta, avg_bits: float, allowed_mask: int, cap: bool = False):
    """Integer allocation as the library defines it: greedy for a contiguous
    allowed set, exact DP otherwise. Returns (bits or None, objective)."""
    w = cap_weights(w) if cap else [float(x) for x in w]
    alpha = [float(x) for x in alpha]
    beta = [float(x) for x in beta]
    n = len(w)
    allowed = allowed_bits(allowed_mask)
    B = budget(avg_bits, n)
    if is_contiguous(allowed):
        bits = greedy(w, alpha, beta, B, allowed[0], allowed[-1])
    else:
        bits = dp(w, alpha, beta, B, allowed)
    if bits is None:
        return None, math.nan
    return bits, objective(w, alpha, beta, bits)


def continuous(w, alpha, beta, avg_bits: float, b_min: float, b_max: float):
    """Continuous reverse waterfilling with iterative clipping (Thm. 1, App. B.1).

    Free components satisfy w_i alpha_i ln(beta_i) beta_i^-b_i = lambda; the
    budget fixes ln lambda in closed form:
      ln lambda = (sum_F A_i / ln beta_i - B_F) / sum_F 1 / ln beta_i,
      A_i = ln(w_i alpha_i ln beta_i).
    Components outside [b_min, b_max] are clipped and fixed; repeat.
    Returns list of floats, or None if avg_bits is outside the bounds.
    """
    n = len(w)
    B = avg_bits * n
    if B < n * b_min - 1e-9 or B > n * b_max + 1e-9:
        return None
    A = [math.log(float(w[i]) * float(alpha[i]) * math.log(float(beta[i]))) for i in range(n)]
    lb = [math.log(float(beta[i])) for i in range(n)]
    fixed = [None] * n
    out = [0.0] * n
    for _ in range(n + 1):
        free = [i for i in range(n) if fixed[i] is None]
        if not free:
            break
        Bf = B
        for i in range(n):
            if fixed[i] is not None:
                Bf -= fixed[i]
        num = 0.0
        den = 0.0
        for i in free:
            num += A[i] / lb[i]
            den += 1.0 / lb[i]
        ln_lam = (num - Bf) / den
        changed = False
        for i in free:
            b = (A[i] - ln_lam) / lb[i]
            if b < b_min:
                fixed[i] = float(b_min)
                changed = True
            elif b > b_max:
                fixed[i] = float(b_max)
                changed = True
            else:
                out[i] = b
        if not changed:
            break
    for i in range(n):
        if fixed[i] is not None:
            out[i] = fixed[i]
    return out


def am_gm(w) -> float:
    n = len(w)
    am = 0.0
    lg = 0.0
    for x in w:
        am += float(x)
        lg += math.log(float(x))
    return (am / n) / math.exp(lg / n)
