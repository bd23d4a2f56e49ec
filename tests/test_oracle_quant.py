"""Pins for the oracle quantizer and rotation (CPU only).

Each test checks the oracle against something other than itself: exact
reconstruction cases, the uniform-quantization noise law s^2/12, the error
bound |x - x_hat| <= s/2, monotonicity in b, and the textbook Sylvester /
scipy Hadamard matrix.
"""
import numpy as np
import pytest
import scipy.linalg

from oracle import quant
from oracle.attention import rotation_matrix, sylvester_hadamard


@pytest.mark.parametrize("b", range(1, 9))
def test_constant_group_is_exact(b):
    # A constant group has zero range: scale 0, every code 0, x_hat = x
    # exactly when the value is representable in fp16 (App. W KIVI kernel,
    # 8-bit case included).
    for val in (0.0, 1.5, -3.25, 1000.0, 2.0 ** -14):
        x = np.full((3, 32), val, dtype=np.float32)
        codes, scale, zero, bad = quant.quantize_groups(x, b)
        assert not bad.any()
        assert (codes == 0).all()
        assert (scale == 0).all()
        xhat = quant.dequantize_groups(codes, scale, zero)
        assert np.array_equal(xhat, x)


def test_integer_group_at_8_bits_is_exact():
    # Values 0..255 in one group of 32 (min 0, max 255): scale = 255/255 = 1,
    # zero = 0, codes equal the values, reconstruction is exact.
    rng = np.random.default_rng(1)
    x = rng.integers(0, 256, size=(64, 32)).astype(np.float32)
    x[:, 0] = 0.0
    x[:, 1] = 255.0
    codes, scale, zero, bad = quant.quantize_groups(x, 8)
    assert (scale == 1.0).all() and (zero == 0.0).all() and not bad.any()
    assert np.array_equal(codes.astype(np.float32), x)
    assert np.array_equal(quant.dequantize_groups(codes, scale, zero), x)


@pytest.mark.parametrize("b", range(1, 9))
def test_error_bound_half_step(b):
    # Asymmetric min-max rounding: |x - x_hat| <= s/2 plus the fp16 rounding
    # of the zero-point and of the scale times the code range.
    rng = np.random.default_rng(b)
    x = rng.standard_normal((2048, 32)).astype(np.float32) * 3.0
    codes, scale, zero, bad = quant.quantize_groups(x, b)
    xhat = quant.dequantize_groups(codes, scale, zero)
    sf = scale.astype(np.float64)[:, None]
    mn = x.min(axis=1, keepdims=True).astype(np.float64)
    zslack = np.abs(zero.astype(np.float64)[:, None] - mn)
    L = 2 ** b - 1
    s_exact = (x.max(axis=1, keepdims=True) - mn) / L
    sslack = L * np.abs(sf - s_exact)
    err = np.abs(x.astype(np.float64) - xhat)
    assert (err <= sf / 2 + zslack + sslack + 1e-6).all()
    assert codes.max() <= L


def test_mse_decreases_with_bits():
    # D(b) strictly decreasing in b on Gaussian groups (Assumption 1, beta > 1).
    rng = np.random.default_rng(7)
    x = rng.standard_normal((65536 // 32 * 32, 32)).astype(np.float32)
    mse = []
    for b in range(1, 9):
        codes, scale, zero, _ = quant.quantize_groups(x, b)
        xhat = quant.dequantize_groups(codes, scale, zero)
        mse.append(np.mean((x.astype(np.float64) - xhat) ** 2))
    assert all(mse[i + 1] < mse[i] for i in range(7)), mse


@pytest.mark.parametrize("b", [2, 4, 6])
def test_uniform_noise_law(b):
    # Uniform data filling [0, 1] with both ends present: the error of a
    # uniform quantizer with step s is uniform on [-s/2, s/2], MSE = s^2/12
    # (textbook high-resolution result). 3-sigma of the estimate ~ 2e-3.
    rng = np.random.default_rng(100 + b)
    n = 65536
    x = rng.random((n, 32)).astype(np.float32)
    x[:, 0] = 0.0
    x[:, 1] = 1.0
    codes, scale, zero, _ = quant.quantize_groups(x, b)
    xhat = quant.dequantize_groups(codes, scale, zero)
    # the two forced endpoints sit on grid points; measure the other 30 columns
    mse = np.mean((x[:, 2:].astype(np.float64) - xhat[:, 2:]) ** 2)
    s = float(scale[0])
    assert (scale == scale[0]).all()
    assert abs(mse / (s * s / 12.0) - 1.0) < 0.01


def test_rounding_is_half_even_and_codes_use_stored_scale():
    # One group, b = 2: values chosen so (x - zero)/scale lands exactly on .5.
    # min 0, max 3 -> scale 1, zero 0; 0.5 -> 0, 1.5 -> 2, 2.5 -> 2 (ties to even).
    x = np.zeros((1, 32), dtype=np.float32)
    x[0, 1] = 3.0
    x[0, 2] = 0.5
    x[0, 3] = 1.5
    x[0, 4] = 2.5
    codes, scale, zero, _ = quant.quantize_groups(x, 2)
    assert scale[0] == 1.0 and zero[0] == 0.0
    assert list(codes[0, :5]) == [0, 3, 0, 2, 2]


def test_negative_zero_is_canonical():
    # -0 and +0 quantize the same way; the stored zero-point is +0.
    x = np.zeros((2, 32), dtype=np.float32)
    x[0, :] = -0.0
    codes, scale, zero, bad = quant.quantize_groups(x, 3)
    assert np.array_equal(zero.view(np.uint16), np.zeros(2, np.uint16))


def test_numeric_failures_are_flagged():
    x = np.zeros((4, 32), dtype=np.float32)
    x[0, 3] = np.nan
    x[1, 5] = np.inf
    x[2, 0] = 1e6           # zero-point or range overflows fp16
    x[2, 1] = -1e6
    x[3, :] = np.arange(32)
    codes, scale, zero, bad = quant.quantize_groups(x, 4)
    assert list(bad) == [True, True, True, False]
    assert (codes[:3] == 0).all() and (scale[:3] == 0).all() and (zero[:3] == 0).all()


def test_grouping_views_round_trip():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((96, 128)).astype(np.float32)
    for gp in (quant.PER_TOKEN, quant.PER_CHANNEL):
        g = quant.to_groups(x, gp)
        assert np.array_equal(quant.from_groups(g, gp), x)
    g = quant.to_groups(x, quant.PER_CHANNEL)
    assert np.array_equal(g[1, 5], x[32:64, 5])          # 32 tokens of channel 5
    g = quant.to_groups(x, quant.PER_TOKEN)
    assert np.array_equal(g[7, 2], x[7, 64:96])          # channels 64..95 of token 7


def test_sylvester_matches_scipy():
    assert np.array_equal(sylvester_hadamard(128), scipy.linalg.hadamard(128))


def test_rotation_orthogonal():
    rng = np.random.default_rng(5)
    signs = rng.choice([-1, 1], size=128).astype(np.int8)
    R = rotation_matrix(signs)
    assert np.allclose(R @ R.T, np.eye(128), atol=1e-12)


def test_fwht_of_unit_vectors_is_hadamard_column():
    # FWHT(e_k)/sqrt(128) is row k of H/sqrt(128) (H symmetric).
    H = scipy.linalg.hadamard(128).astype(np.float64) / np.sqrt(128)
    E = np.eye(128, dtype=np.float32)
    Y = quant.hadamard_rotate(E, None).astype(np.float64)
    assert np.allclose(Y, H, rtol=1e-7, atol=0)


def test_fwht_matches_matrix_product():
    rng = np.random.default_rng(9)
    signs = rng.choice([-1, 1], size=128).astype(np.int8)
    x = rng.standard_normal((200, 128)).astype(np.float32)
    y = quant.hadamard_rotate(x, signs).astype(np.float64)
    ref = x.astype(np.float64) @ (np.diag(signs.astype(np.float64))
                                  @ scipy.linalg.hadamard(128) / np.sqrt(128))
    assert np.allclose(y, ref, rtol=0, atol=1e-5 * np.abs(ref).max())


def test_rotation_preserves_mse():
    # R orthogonal: the error measured in the rotated domain equals the error
    # after rotating back, up to fp32/fp64 rounding.
    rng = np.random.default_rng(11)
    signs = rng.choice([-1, 1], size=128).astype(np.int8)
    x = rng.standard_normal((256, 128)).astype(np.float32)
    r = quant.quantize_stream(x, quant.PER_TOKEN, 4, signs, hadamard=True)
    e_rot = np.mean((r["y"].astype(np.float64) - r["xhat"]) ** 2)
    R = rotation_matrix(signs)
    back = r["xhat"].astype(np.float64) @ R.T
    e_orig = np.mean((x.astype(np.float64) - back) ** 2)
    assert abs(e_rot / e_orig - 1.0) < 1e-5


def _round_half_even(fr):
    from fractions import Fraction
    lo = fr.numerator // fr.denominator
    rem = fr - lo
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and lo % 2 == 1):
        return lo + 1
    return lo


@pytest.mark.parametrize("b", (2, 3, 4, 8))
def test_codes_are_exact_rational_rounding(b):
    # code = clamp(round_half_even((fp32(v - zf)) * inv), 0, L) with the product
    # taken exactly: checked with rational arithmetic, element by element.
    from fractions import Fraction
    rng = np.random.default_rng(100 + b)
    x = (rng.standard_normal((40, 32)) * rng.uniform(0.01, 50, (40, 1))).astype(np.float32)
    codes, scale, zero, bad = quant.quantize_groups(x, b)
    L = 2 ** b - 1
    for g in range(x.shape[0]):
        sf = np.float32(scale[g])
        zf = np.float32(zero[g])
        inv = np.float32(1.0) / sf
        for j in range(32):
            d = np.float32(np.float32(x[g, j]) - zf)
            want = min(max(_round_half_even(Fraction(float(d)) * Fraction(float(inv))), 0), L)
            assert codes[g, j] == want


def test_one_rounding_not_two():
    # A value v whose exact product v * inv lies just below k + 1/2 while its
    # fp32 rounding is exactly k + 1/2 (k odd): rounding the fp32 product
    # would give the even neighbour k + 1, the exact product gives k. The
    # group min 0, max m at b = 8 fixes scale = fp16(m / 255), zero = 0.
    from fractions import Fraction
    b = 8
    found = None
    for m in range(3, 200):
        sf = np.float32(np.float16(np.float32(m) / np.float32(255.0)))
        inv = np.float32(1.0) / sf
        for k in range(1, 255, 2):
            half = Fraction(2 * k + 1, 2)
            v = np.float32(float(half / Fraction(float(inv))))
            cands = [v]
            lo = hi = v
            for _ in range(3):
                lo = np.nextafter(lo, np.float32(-1e9))
                hi = np.nextafter(hi, np.float32(1e9))
                cands += [lo, hi]
            for cand in cands:
                exact = Fraction(float(cand)) * Fraction(float(inv))
                fp32_product = float(np.float32(float(cand) * float(inv)))   # fp64 product is exact
                if exact < half and fp32_product == k + 0.5 and 0 < cand < m:
                    found = (m, k, np.float32(cand))
                    break
            if found:
                break
        if found:
            break
    assert found is not None
    m, k, v = found
    x = np.zeros((1, 32), dtype=np.float32)
    x[0, 1] = np.float32(m)
    x[0, 2] = v
    codes, scale, zero, _ = quant.quantize_groups(x, b)
    assert float(zero[0]) == 0.0
    assert codes[0, 2] == k


def test_symmetric_levels_are_exact():
    # b = 3 (M = 3), a = 3 * 2^-2: levels q / 4, q = -3..3 (scale 2^-2 and
    # zero -3/4 both exact in fp16), code q + 3; a group drawn from the levels
    # with +a present reconstructs exactly, and its min does not matter
    rng = np.random.default_rng(21)
    lv = np.arange(-3, 4, dtype=np.float32) / 4
    x = lv[rng.integers(0, 7, size=(50, 32))]
    x[:, 0] = 0.75
    x[:, 1] = 0.25
    x[x < -0.5] = 0.0
    codes, scale, zero, bad = quant.quantize_groups(x, 3, symmetric=True)
    assert (scale == 0.25).all() and (zero == -0.75).all() and not bad.any()
    assert np.array_equal(codes.astype(np.float32), 4 * x + 3)
    assert np.array_equal(quant.dequantize_groups(codes, scale, zero), x)
    assert codes.max() <= 6                       # code 2^b - 1 is never used


def test_symmetric_matches_printed_absmax_formula():
    # round(x M / a) a / M (App. W, "TurboQuant kernel") in exact arithmetic,
    # when a / M is a power of two (scale and zero exact in fp16) and no value
    # sits on a rounding tie
    rng = np.random.default_rng(22)
    for b in range(2, 9):
        M = 2 ** (b - 1) - 1
        for e in (-6, 0, 3):
            a = M * 2.0 ** e
            x = rng.uniform(-a, a, size=(64, 32))
            x[:, 5] = -a if b % 2 else a
            x = x.astype(np.float16).astype(np.float32)
            u = x.astype(np.float64) * M / a
            keep = np.abs(u - np.floor(u) - 0.5) > 1e-9
            codes, scale, zero, bad = quant.quantize_groups(x, b, symmetric=True)
            assert not bad.any() and (scale == 2.0 ** e).all()
            want = np.round(u) * a / M
            got = quant.dequantize_groups(codes, scale, zero).astype(np.float64)
            assert np.array_equal(got[keep], want[keep]), (b, e)
            assert np.array_equal((codes.astype(np.int64) - M)[keep], np.round(u).astype(np.int64)[keep])


def test_symmetric_one_bit_has_the_single_level_zero():
    # M = 2^0 - 1 = 0: the absmax form has one level, 0
    x = np.random.default_rng(23).standard_normal((40, 32)).astype(np.float32)
    codes, scale, zero, bad = quant.quantize_groups(x, 1, symmetric=True)
    assert not bad.any() and (codes == 0).all() and (scale == 0).all() and (zero == 0).all()
    assert (zero.view(np.uint16) == 0).all()      # +0, not -0: the stored words are exact
    assert (quant.dequantize_groups(codes, scale, zero) == 0).all()


@pytest.mark.parametrize("b", range(2, 9))
def test_symmetric_codes_are_nearest_level(b):
    # brute force over every code: the chosen level is the nearest one of the
    # 2M + 1 stored levels (up to the fp32 rounding of x - zero near a tie)
    rng = np.random.default_rng(40 + b)
    x = (rng.standard_normal((256, 32)) * np.exp(rng.uniform(-4, 4, (256, 1)))).astype(np.float32)
    codes, scale, zero, bad = quant.quantize_groups(x, b, symmetric=True)
    assert not bad.any()
    M = 2 ** (b - 1) - 1
    sf = scale.astype(np.float64)[:, None, None]
    zf = zero.astype(np.float64)[:, None, None]
    levels = np.arange(2 * M + 1)[None, None, :] * sf + zf
    dist = np.abs(x.astype(np.float64)[..., None] - levels)
    best = dist.min(axis=-1)
    mine = np.take_along_axis(dist, codes[..., None].astype(np.int64), axis=-1)[..., 0]
    a = np.abs(x).max(axis=-1, keepdims=True).astype(np.float64)
    assert (mine <= best + 2.0 ** -22 * a).all()      # the fp32 rounding of x - zero
    # mirror symmetry of the levels about 0, up to the fp16 rounding of zero
    assert (np.abs(zf[..., 0] + M * sf[..., 0]) <= 2.0 ** -11 * np.abs(zf[..., 0])).all()


@pytest.mark.parametrize("b", range(2, 9))
def test_symmetric_error_bound(b):
    # |x - x_hat| <= s / 2 + the fp16 rounding of zero, s = max|x| / M
    rng = np.random.default_rng(30 + b)
    x = rng.standard_normal((1024, 32)).astype(np.float32) * 2.0
    codes, scale, zero, bad = quant.quantize_groups(x, b, symmetric=True)
    xhat = quant.dequantize_groups(codes, scale, zero).astype(np.float64)
    M = 2 ** (b - 1) - 1
    sf = scale.astype(np.float64)[:, None]
    zslack = np.abs(zero.astype(np.float64)[:, None] + M * sf)
    a = np.abs(x).max(axis=1, keepdims=True).astype(np.float64)
    assert (np.abs(x - xhat) <= sf / 2 + zslack + 1e-6 * a).all()
    assert (np.abs(sf - a / M) <= 2.0 ** -11 * a / M).all()


def test_symmetric_costs_one_level():
    # the absmax form spends one code (2M + 1 = 2^b - 1 levels over a range
    # 2a >= max - min), so on the same data its MSE is never far below the
    # min-max form's and, for zero-mean data, about (2^b - 1)^2 / (2^b - 2)^2
    # times it: a different beta, the point of a per-quantizer calibration
    rng = np.random.default_rng(24)
    x = rng.standard_normal((4096, 32)).astype(np.float32)
    for b in (3, 4, 6):
        ms = []
        for sym in (False, True):
            c, s, z, _ = quant.quantize_groups(x, b, symmetric=sym)
            ms.append(((quant.dequantize_groups(c, s, z) - x) ** 2).mean())
        assert ms[1] > ms[0]


# ---- TurboQuant group sizes (App. W "TurboQuant kernel": absmax per group,
# 128 elements for keys, 64 for values, along one token's head dimension)

def test_wide_groups_match_printed_absmax_formula():
    # round(x M / a) a / M with a = max |x| over each group of 128 (one key
    # row) or 64 (half a value row), when a / M is a power of two and no value
    # sits on a tie
    rng = np.random.default_rng(31)
    for grouping, n in ((quant.PER_TOKEN_128, 128), (quant.PER_TOKEN_64, 64)):
        for b in (2, 3, 4, 8):
            M = 2 ** (b - 1) - 1
            e = rng.integers(-4, 4, size=(48, 128 // n))          # a / M = 2^e per group
            a = M * 2.0 ** e
            x = rng.uniform(-1, 1, size=(48, 128 // n, n)) * a[..., None]
            x[:, :, 7] = a                                       # the group's absmax
            x = x.astype(np.float16).astype(np.float32).reshape(48, 128)
            u = (x.reshape(48, 128 // n, n).astype(np.float64) * M / a[..., None]).reshape(48, 128)
            keep = np.abs(u - np.floor(u) - 0.5) > 1e-9
            r = quant.quantize_stream(x, grouping, b, symmetric=quant.ABSMAX)
            assert (r["group_scale"] == 2.0 ** e).all() and not r["bad"].any()
            want = np.round(u) * np.repeat(a / M, n, axis=1)
            got = r["xhat"].astype(np.float64)
            assert np.array_equal(got[keep], want[keep]), (n, b)
            assert np.array_equal((r["codes"].astype(np.int64) - M)[keep], np.round(u).astype(np.int64)[keep])


def test_wide_groups_store_their_parameters_on_every_group_of_32():
    # a key row of 128 with absmax 14 at 4 bits: scale 2, zero -14 on all four
    # stored groups of 32; a value row whose halves have absmax 14 and 7:
    # scales 2, 2, 1, 1 and zeros -14, -14, -7, -7
    x = np.zeros((32, 128), dtype=np.float32)
    x[:, 3] = 14.0
    x[:, 100] = -6.0
    r = quant.quantize_stream(x, quant.PER_TOKEN_128, 4, symmetric=quant.ABSMAX)
    assert r["scale"].shape == (32, 4) and (r["scale"] == 2.0).all() and (r["zero"] == -14.0).all()
    assert (r["group_scale"].shape == (32, 1))
    assert (r["codes"][:, 3] == 14).all() and (r["codes"][:, 100] == 4).all() and (r["codes"][:, 0] == 7).all()
    y = np.zeros((32, 128), dtype=np.float32)
    y[:, 10] = -14.0
    y[:, 64 + 20] = 7.0
    r = quant.quantize_stream(y, quant.PER_TOKEN_64, 4, symmetric=quant.ABSMAX)
    assert (r["scale"] == np.float16([2, 2, 1, 1])).all() and (r["zero"] == np.float16([-14, -14, -7, -7])).all()
    assert (r["codes"][:, 10] == 0).all() and (r["codes"][:, 84] == 14).all()


def test_wide_groups_equal_groups_of_32_when_their_quarters_agree():
    # every group of 32 of a row holding the same absmax: the wide group's
    # parameters are the same as each quarter's, so the codes agree
    rng = np.random.default_rng(33)
    x = rng.standard_normal((64, 128)).astype(np.float16).astype(np.float32)
    x[:, [0, 32, 64, 96]] = 5.0
    r32 = quant.quantize_stream(x, quant.PER_TOKEN, 3, symmetric=quant.ABSMAX)
    for g in (quant.PER_TOKEN_64, quant.PER_TOKEN_128):
        r = quant.quantize_stream(x, g, 3, symmetric=quant.ABSMAX)
        assert np.array_equal(r["codes"], r32["codes"]) and np.array_equal(r["scale"], r32["scale"])


def test_wider_groups_cost_distortion():
    # on Gaussian rows a larger group has a larger absmax, so a coarser step:
    # MSE(128) > MSE(64) > MSE(32) at every width (statistical, 4096 tokens)
    x = np.random.default_rng(34).standard_normal((4096, 128)).astype(np.float32)
    for b in (2, 3, 4, 6):
        mse = []
        for g in (quant.PER_TOKEN, quant.PER_TOKEN_64, quant.PER_TOKEN_128):
            r = quant.quantize_stream(x, g, b, symmetric=quant.ABSMAX)
            mse.append(float(np.mean((r["y"].astype(np.float64) - r["xhat"]) ** 2)))
        assert mse[0] < mse[1] < mse[2], (b, mse)
