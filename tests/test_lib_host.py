"""librq host half on the CPU: the library builds, loads and exports every
symbol include/rq.h declares; its host functions (fit, allocation, layout)
agree with the oracle on identical inputs. No CUDA compute is launched."""
import math
import os
import re

import numpy as np
import pytest

from oracle import alloc as oalloc
from oracle import calib as ocalib
from oracle import pack as opack

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="session")
def rq():
    from paper_2605_06675_gb300 import build, rq as binding
    srcs = [os.path.join(build.CSRC, f) for f in os.listdir(build.CSRC)]
    srcs.append(os.path.join(build.INCLUDE, "rq.h"))
    if not os.path.exists(build.LIB) or os.path.getmtime(build.LIB) < max(map(os.path.getmtime, srcs)):
        build.build()
    binding.lib()
    return binding


def test_exports_every_header_symbol(rq):
    header = open(os.path.join(ROOT, "include", "rq.h")).read()
    declared = sorted(set(re.findall(r"\b(rq_[a-z_]+)\s*\(", header)))
    assert declared, "no declarations found"
    lib = rq.lib()
    for name in declared:
        assert hasattr(lib, name), name
    assert sorted(rq.EXPORTS) == declared
    assert rq.rq_abi_version() == 2
    assert rq.rq_status_string(3) == "unsupported shape"


def test_decode_pattern_setting(rq):
    # host-only: the two documented values are accepted, any other refused
    lib = rq.lib()
    assert lib.rq_decode_set_pattern(rq.RQ_DECODE_INTERLEAVED) == rq.RQ_OK
    assert lib.rq_decode_set_pattern(rq.RQ_DECODE_BACK_TO_BACK) == rq.RQ_OK
    for bad in (-1, 2, 7):
        assert rq.STATUS_NAMES[lib.rq_decode_set_pattern(bad)] == "RQ_ERR_INVALID_ARG"


def _mse_rows(rng, n):
    a = rng.uniform(0.5, 20, n)
    beta = rng.uniform(3.5, 6.0, n)
    b = np.arange(1, 9)
    mse = a[:, None] * beta[:, None] ** (-b[None, :])
    return mse * np.exp(rng.normal(0, 0.05, mse.shape))


def test_fit_matches_oracle(rq):
    rng = np.random.default_rng(0)
    n = 64
    mse = _mse_rows(rng, n)
    mse[3] = [1.0, 0.9, 1e-3, 1e-2, 1e-6, 1e-5, 1e-9, 1e-9]     # poor fit -> fallback
    mse[5] = 0.0                                                 # degenerate
    classes = np.arange(n) % 2
    for lo, hi, r2min in ((2, 6, 0.96), (1, 8, 0.96), (2, 6, 0.0)):
        a, b, r2 = rq.rq_fit_distortion(mse, lo, hi, r2min, classes)
        oa, ob, or2 = ocalib.fit_distortion(mse, lo, hi, r2min, classes)
        assert np.array_equal(a, oa) and np.array_equal(b, ob) and np.array_equal(r2, or2)
    assert rq.rq_fit_distortion(mse, 2, 6, 0.96, None)[1].shape == (n,)


def test_table8_through_the_library(rq):
    # the paper's Table 8 fit (alpha ~ 1.36, beta ~ 3.48) through the C ABI
    row = np.zeros((1, 8))
    row[0, :6] = [3.634e-01, 1.175e-01, 3.455e-02, 9.501e-03, 2.512e-03, 7.647e-04]
    a, b, r2 = rq.rq_fit_distortion(row, 1, 6, 0.0)
    assert abs(a[0] - 1.36) < 0.005 and abs(b[0] - 3.48) < 0.005 and r2[0] > 0.99


@pytest.mark.parametrize("allowed,avg", [((2, 3, 4), 2.5), ((2, 3, 4), 3.0),
                                         ((2, 3, 4, 5, 6, 7, 8), 4.0), ((2, 3, 4, 8), 3.0),
                                         ((1, 2, 3, 4, 5, 6, 7, 8), 3.3), ((2, 8), 4.0)])
def test_alloc_matches_oracle(rq, allowed, avg):
    rng = np.random.default_rng(int(avg * 10) + len(allowed))
    n = 96
    w = np.exp(rng.normal(0, 0.76, n))
    a = rng.uniform(0.5, 20, n)
    beta = rng.uniform(3.5, 6.0, n)
    mask = sum(1 << k for k in allowed)
    for cap in (False, True):
        bits, J = rq.rq_alloc(w, a, beta, avg, mask, rq.RQ_CAP_5X if cap else 0)
        obits, oJ = oalloc.allocate(w, a, beta, avg, mask, cap)
        assert obits is not None
        assert list(bits) == obits
        assert J == oJ
        assert int(bits.sum()) == oalloc.budget(avg, n)


def test_alloc_ties_and_errors(rq):
    n = 10
    bits, _ = rq.rq_alloc([1.0] * n, [1.0] * n, [4.0] * n, 3.4, 0b1111100)
    assert list(bits) == [4, 4, 4, 4, 3, 3, 3, 3, 3, 3]
    with pytest.raises(rq.RQError) as e:
        rq.rq_alloc([1.0] * 3, [1.0] * 3, [4.0] * 3, 7.0 / 3.0, (1 << 2) | (1 << 8))
    assert e.value.status == 2            # 7 bits over {2, 8} is unreachable
    with pytest.raises(rq.RQError) as e:
        rq.rq_alloc([1.0] * 3, [1.0] * 3, [4.0] * 3, 3.0, 1)       # bit 0 is not a width
    assert e.value.status == 1


def test_continuous_matches_oracle(rq):
    rng = np.random.default_rng(3)
    n = 80
    w = np.exp(rng.normal(0, 1.2, n))
    a = rng.uniform(1, 10, n)
    beta = rng.uniform(3.5, 5.5, n)
    for lo, hi, avg in ((2.0, 4.0, 3.0), (0.0, 16.0, 4.0), (3.0, 6.0, 4.5)):
        got = rq.rq_alloc_continuous(w, a, beta, avg, lo, hi)
        ref = oalloc.continuous(list(w), list(a), list(beta), avg, lo, hi)
        assert np.array_equal(got, np.array(ref))
        assert abs(got.sum() - avg * n) < 1e-8
    with pytest.raises(rq.RQError):
        rq.rq_alloc_continuous(w, a, beta, 5.0, 2.0, 4.0)


def test_packed_layout_matches_oracle(rq):
    rng = np.random.default_rng(4)
    L, B, H, S = 3, 2, 4, 96
    bits = rng.integers(1, 9, size=(L, H, 2)).astype(np.uint8)
    desc = rq.make_desc(L, B, H, 4 * H, S, rq.RQ_BF16, rq.RQ_PER_CHANNEL, rq.RQ_PER_TOKEN)
    off, total = rq.rq_packed_layout(desc, bits)
    ooff, ototal = opack.stream_offsets(L, B, H, S, bits)
    assert total == ototal and np.array_equal(off, ooff)
    assert all(int(o) % 512 == 0 for o in off.reshape(-1))
    bad = rq.make_desc(L, B, H, 4 * H, 100, rq.RQ_BF16, 1, 0)
    with pytest.raises(rq.RQError) as e:
        rq.rq_packed_layout(bad, bits)
    assert e.value.status == 3
    bits[0, 0, 0] = 9
    with pytest.raises(rq.RQError):
        rq.rq_packed_layout(desc, bits)


DIV_CHECK_C = r"""
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>
/* The quantizer's scale division: q0 = RN(x yi), r = RN(x - q0 y) by one fma,
   q = RN(q0 + r yi), yi = RN(1 / y), against x / y, for every significand of x
   in [1, 2) and y = 2^k - 1, k = 1..8. */
int main(void) {
  long bad = 0;
  for (int k = 1; k <= 8; ++k) {
    const float y = (float)((1 << k) - 1), yi = 1.0f / y;
    for (uint32_t m = 0; m < (1u << 23); ++m) {
      uint32_t u = (127u << 23) | m;
      float x;
      memcpy(&x, &u, 4);
      const float q0 = x * yi;
      const float r = fmaf(-q0, y, x);
      const float q = fmaf(r, yi, q0);
      if (q != x / y) ++bad;
    }
  }
  printf("%ld\n", bad);
  return 0;
}
"""


def test_scale_division_method_is_exact(tmp_path):
    # The kernels divide the group range by 2^b - 1 (and the absmax by
    # 2^(b-1) - 1) with a correction step instead of an IEEE division; this
    # proves it exact for every fp32 significand on an IEEE host (binary32
    # multiply and fma correctly rounded, no contraction).
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "div.c"
    src.write_text(DIV_CHECK_C)
    exe = tmp_path / "div"
    subprocess.run([cc, "-O2", "-ffp-contract=off", "-o", str(exe), str(src), "-lm"], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    assert out.strip() == "0"


def test_lloydmax_codebook_matches_the_oracle(rq):
    # the library solves the codebook on its own (C++, upper half, Newton);
    # its fp16 levels must equal the oracle's at every width
    from oracle import lloydmax
    for b in range(1, 9):
        got = rq.rq_lloydmax_levels(b)
        want = lloydmax.levels_f16(b)
        assert np.array_equal(got.view(np.uint16), want.view(np.uint16)), b
    with pytest.raises(rq.RQError):
        rq.rq_lloydmax_levels(9)


def test_lloydmax_midpoints_fit_the_quantizer_buckets(rq):
    """The quantize kernel finds a Lloyd-Max code from a bucket of u = v / scale
    (1024 equal bins over [-5, 5)) and one exact threshold comparison; that is
    exact only if no bin widened by 1e-5 on each side holds more than one of the
    codebook's fp32 midpoints and none lies in the end bins. Checked here on
    the library's own codebooks, every width."""
    bins, r, delta = 1024, 5.0, 1e-5
    w = 2 * r / bins
    assert w == 0.009765625                        # the kernel's exact bin step
    for b in range(1, 9):
        lv = rq.rq_lloydmax_levels(b).view(np.float16).astype(np.float32)
        mid = ((lv[:-1] + lv[1:]) * np.float32(0.5)).astype(np.float64)
        assert np.all(np.abs(mid) < r - w), b
        for k in range(bins):
            lo, hi = -r + k * w - delta, -r + (k + 1) * w + delta
            assert int(((mid >= lo) & (mid < hi)).sum()) <= 1, (b, k)
