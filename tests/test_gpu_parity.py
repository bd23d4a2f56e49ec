"""GPU parity: librq (through the C ABI) against the CPU oracle on the same
seeded inputs. Codes, scales, zero-points and packed words bit-exact;
attention within 2e-3 * max(1, max|o|); MSE sweep within 1e-9 relative."""
import numpy as np
import pytest
import torch

from oracle import calib as ocalib
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import (PER_CHANNEL, PER_TOKEN, PER_TOKEN_64, PER_TOKEN_128,
                                              Workload)

from .gpu_helpers import (TOL, attn_err, bits_cycle, ensure_built, oracle_attention,
                          oracle_layer, to_np)

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def rq():
    return ensure_built()


def small_wl(L=2, B=2, H=4, g=4, S=96, dtype="float16", kg=PER_CHANNEL, vg=PER_TOKEN,
             hadamard=False, seed=11, value_dist="gaussian", kq=0, vq=0):
    return Workload(f"t{seed}", L=L, B=B, H_kv=H, H_q=H * g, S=S, dtype=dtype, k_grouping=kg,
                    v_grouping=vg, hadamard=hadamard, allowed=tuple(range(1, 9)), avg_bits=4.0,
                    sigma_lnw=0.5, value_dist=value_dist, seed=seed, k_quantizer=kq,
                    v_quantizer=vq)


def symmetric_of(wl):
    """The oracle's quantizer forms (0 min-max, 1 absmax, 2 Lloyd-Max) of K and V."""
    return (int(wl.k_quantizer), int(wl.v_quantizer))


def run_layers(rq, wl, bits, layers=None, q_seed=0, kv_scale=1.0):
    """Quantize every layer and decode; returns (path, {l: (k, v, q, out)})."""
    signs = synth.hadamard_signs(wl.seed) if wl.hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    path.set_bits(bits)
    res = {}
    for l in (range(wl.L) if layers is None else layers):
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, wl.value_dist, DEV)
        if kv_scale != 1.0:
            k, v = k * kv_scale, v * kv_scale
        q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed + q_seed, l, DEV)
        out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
        path.quantize(l, k, v)
        path.decode(l, q, out)
        res[l] = (k, v, q, out)
    torch.cuda.synchronize()
    return path, res, signs


def check_layer(path, wl, l, k, v, q, out, signs, streams=None):
    """Bit-exact packed bytes and attention within TOL for the given streams."""
    ol = oracle_layer(k, v, path.bits_host[l], wl.k_grouping, wl.v_grouping, wl.hadamard,
                      signs, streams, symmetric_of(wl))
    for (bb, h, kind), r in ol.items():
        got = path.stream_bytes(l, bb, h, kind).cpu().numpy()
        want = r["words"].view(np.uint8)
        assert got.shape == want.shape
        if not np.array_equal(got, want):
            nbad = int((got != want).sum())
            raise AssertionError(f"layer {l} stream ({bb},{h},{kind}) b={path.bits_host[l, h, kind]}: "
                                 f"{nbad} of {got.size} bytes differ")
    ref = oracle_attention(q, ol, wl.g)
    keys = sorted(ref)
    got = to_np(out)
    err = attn_err(np.stack([got[bb, j] for bb, j in keys]), np.stack([ref[key] for key in keys]))
    assert err <= TOL, f"layer {l}: attention error {err:.3e}"
    return err


@pytest.mark.parametrize("dtype", ["float16", "bfloat16"])
@pytest.mark.parametrize("kg,vg", [(PER_CHANNEL, PER_TOKEN), (PER_TOKEN, PER_TOKEN),
                                   (PER_TOKEN, PER_CHANNEL), (PER_CHANNEL, PER_CHANNEL)])
def test_all_widths_bit_exact_and_attention(rq, dtype, kg, vg):
    wl = small_wl(dtype=dtype, kg=kg, vg=vg, S=96)
    bits = bits_cycle(wl.L, wl.H_kv, range(1, 9))
    path, res, signs = run_layers(rq, wl, bits)
    for l, (k, v, q, out) in res.items():
        check_layer(path, wl, l, k, v, q, out, signs)
    assert int(path.status.item()) == 0


@pytest.mark.parametrize("dtype", ["float16", "bfloat16"])
def test_hadamard_bit_exact_and_attention(rq, dtype):
    wl = small_wl(dtype=dtype, kg=PER_TOKEN, vg=PER_TOKEN, hadamard=True, S=128, seed=12)
    bits = bits_cycle(wl.L, wl.H_kv, range(1, 9), offset=3)
    path, res, signs = run_layers(rq, wl, bits)
    for l, (k, v, q, out) in res.items():
        check_layer(path, wl, l, k, v, q, out, signs)


@pytest.mark.parametrize("g,H,B,S", [(1, 2, 3, 32), (8, 2, 1, 1024), (3, 2, 2, 32 * 37),
                                     (4, 8, 1, 1024), (8, 1, 1, 32 * 301)])
def test_shapes_gqa_and_splits(rq, g, H, B, S):
    # single block, GQA 1/3/8, odd block counts (ragged splits), long-ish S
    wl = small_wl(L=1, B=B, H=H, g=g, S=S, dtype="bfloat16", seed=13 + g)
    bits = bits_cycle(1, H, (2, 3, 4, 8), offset=g)
    path, res, signs = run_layers(rq, wl, bits)
    k, v, q, out = res[0]
    check_layer(path, wl, 0, k, v, q, out, signs)


def test_heavy_tailed_values(rq):
    wl = small_wl(L=1, B=1, H=2, g=8, S=512, dtype="bfloat16", value_dist="student_t4", seed=21)
    bits = bits_cycle(1, 2, (2, 3, 4, 8))
    path, res, signs = run_layers(rq, wl, bits)
    check_layer(path, wl, 0, *res[0], signs)


def test_constant_and_integer_cache_is_exact(rq):
    # constant K groups and integer V at 8 bits dequantize exactly, so the
    # GPU output equals attention on the original cache (up to fp32 rounding)
    wl = small_wl(L=1, B=1, H=2, g=4, S=64, dtype="float16", seed=23)
    bits = np.full((1, 2, 2), 8, dtype=np.uint8)
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits)
    k = torch.full((1, 2, 64, 128), 0.5, dtype=torch.float16, device=DEV)
    v = torch.randint(0, 256, (1, 2, 64, 128), device=DEV).to(torch.float16)
    v[..., 0::32] = 0
    v[..., 1::32] = 255
    q = synth.queries(1, 8, "float16", 5, 0, DEV)
    out = torch.empty((1, 8, 128), dtype=torch.float32, device=DEV)
    path.quantize(0, k, v)
    path.decode(0, q, out)
    torch.cuda.synchronize()
    want = to_np(v)[0].mean(axis=1)            # equal keys -> mean of V
    got = to_np(out)[0]
    for j in range(8):
        assert np.abs(got[j] - want[j // 4]).max() < 1e-3 * 255


def test_numeric_and_bad_bits_status(rq):
    wl = small_wl(L=1, B=1, H=2, g=4, S=64, dtype="bfloat16", seed=24)
    bits = np.full((1, 2, 2), 4, dtype=np.uint8)
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits)
    k, v = synth.kv_layer(1, 2, 64, "bfloat16", 24, 0, device=DEV)
    k[0, 1, 5, 7] = float("nan")
    path.quantize(0, k, v)
    torch.cuda.synchronize()
    assert int(path.status.item()) & 1          # RQ_STATUS_NUMERIC
    # the other streams are untouched by the NaN group
    ol = oracle_layer(k, v, bits[0], wl.k_grouping, wl.v_grouping, False, None,
                      streams=[(0, 0)])
    assert np.array_equal(path.stream_bytes(0, 0, 0, 0).cpu().numpy(),
                          ol[(0, 0, 0)]["words"].view(np.uint8))
    # a corrupted device bit table is reported, the stream skipped
    path.status.zero_()
    path.bits[0, 0, 1] = 0
    path.quantize(0, k, v)
    q = synth.queries(1, 8, "bfloat16", 1, 0, DEV)
    out = torch.empty((1, 8, 128), dtype=torch.float32, device=DEV)
    path.decode(0, q, out)
    torch.cuda.synchronize()
    assert int(path.status.item()) & 2          # RQ_STATUS_BAD_BITS
    assert torch.isfinite(out).all()


def test_argument_errors(rq):
    wl = small_wl(L=1, B=1, H=2, g=4, S=64, dtype="bfloat16", seed=25)
    path = PackedKVPath(wl, DEV)
    path.set_bits(np.full((1, 2, 2), 3, dtype=np.uint8))
    k, v = synth.kv_layer(1, 2, 64, "bfloat16", 25, 0, device=DEV)
    q = synth.queries(1, 8, "bfloat16", 25, 0, DEV)
    out = torch.empty((1, 8, 128), dtype=torch.float32, device=DEV)
    ws = path.decode_workspace()
    d = path.desc
    bad = rq.make_desc(1, 1, 2, 8, 48, torch.bfloat16, 1, 0)
    with pytest.raises(rq.RQError) as e:
        rq.rq_quantize_pack(bad, 0, k, v, None, path.bits, path.offsets, path.packed)
    assert e.value.status == 3                  # S % 32
    bad = rq.make_desc(1, 1, 2, 18, 64, torch.bfloat16, 1, 0)
    with pytest.raises(rq.RQError) as e:
        rq.rq_decode_attention(bad, 0, q, path.packed, path.bits, path.offsets, None, out, ws)
    assert e.value.status == 3                  # GQA group 9 > 8
    with pytest.raises(rq.RQError) as e:
        rq.rq_quantize_pack(d, 0, k, v, None, path.bits, path.offsets, path.packed[1:])
    assert e.value.status == 4                  # misaligned packed pointer
    with pytest.raises(rq.RQError) as e:
        rq.rq_decode_attention(d, 0, q, path.packed, path.bits, path.offsets, None, out, ws[:16])
    assert e.value.status == 5                  # workspace too small
    with pytest.raises(rq.RQError) as e:
        rq.rq_decode_attention(d, 1, q, path.packed, path.bits, path.offsets, None, out, ws)
    assert e.value.status == 1                  # layer out of range
    empty = rq.make_desc(1, 0, 2, 8, 64, torch.bfloat16, 1, 0)
    rq.rq_quantize_pack(empty, 0, k, v, None, path.bits, path.offsets, path.packed)   # B = 0: no-op


# Tolerance of the MSE sweep, from the arithmetic: per element the GPU forms
# e = fp32(y - y_hat) (relative error <= 2^-24) and accumulates e*e with fp32
# FMAs in two interleaved partial sums of 16 terms each (<= 16 * 2^-24
# relative), then sums groups in fp64. The oracle sums exact fp64 squares.
# Worst case ~1.1e-6 relative per group; 1e-5 leaves a 9x margin.
MSE_RTOL = 1e-5


@pytest.mark.parametrize("hadamard", [False, True])
@pytest.mark.parametrize("dtype", ["bfloat16", "float16"])
def test_calibration_sweep_matches_oracle(rq, hadamard, dtype):
    wl = small_wl(L=2, H=4, S=96, dtype=dtype, hadamard=hadamard, seed=31,
                  kg=PER_TOKEN if hadamard else PER_CHANNEL)
    x = synth.calibration_sample(wl, T=96, device=DEV)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    mse = path.calibrate(x).cpu().numpy()
    torch.cuda.synchronize()
    groupings = [wl.k_grouping if i % 2 == 0 else wl.v_grouping for i in range(x.shape[0])]
    ref = ocalib.distortion_sweep(to_np(x), groupings, hadamard,
                                  None if signs is None else signs.numpy())
    rel = np.abs(mse - ref) / np.abs(ref)
    assert rel.max() < MSE_RTOL, rel.max()
    assert np.all(np.diff(mse, axis=1) < 0)


def test_calibration_rotated_per_channel(rq):
    # rotation with per-channel groups regroups the rotated tile by column
    wl = small_wl(L=1, H=4, S=64, dtype="bfloat16", hadamard=True, seed=33,
                  kg=PER_CHANNEL, vg=PER_CHANNEL)
    x = synth.calibration_sample(wl, T=64, device=DEV)
    signs = synth.hadamard_signs(wl.seed)
    path = PackedKVPath(wl, DEV, signs)
    mse = path.calibrate(x).cpu().numpy()
    ref = ocalib.distortion_sweep(to_np(x), [PER_CHANNEL] * x.shape[0], True, signs.numpy())
    assert (np.abs(mse - ref) / ref).max() < MSE_RTOL


def test_hadamard_per_channel_bit_exact(rq):
    wl = small_wl(L=1, B=2, H=2, g=4, S=64, dtype="bfloat16", kg=PER_CHANNEL, vg=PER_CHANNEL,
                  hadamard=True, seed=34)
    bits = bits_cycle(1, 2, range(1, 9), offset=5)
    path, res, signs = run_layers(rq, wl, bits)
    check_layer(path, wl, 0, *res[0], signs)


def test_calibration_deterministic(rq):
    wl = small_wl(L=1, H=8, dtype="bfloat16", seed=32)
    x = synth.calibration_sample(wl, T=512, device=DEV)
    path = PackedKVPath(wl, DEV)
    a = path.calibrate(x).clone()
    b = path.calibrate(x).clone()
    assert torch.equal(a, b)


# ---- symmetric absmax quantizer (App. W "TurboQuant kernel" form) -----------
# KIVI: per-channel symmetric keys, per-token asymmetric values (Sec. 2);
# RTN: per-token symmetric (Table 16); QuaRot: rotation + per-token
# symmetric (Sec. 4.1); and every grouping with both kinds symmetric.
SYM_CASES = [
    ("kivi", "float16", PER_CHANNEL, PER_TOKEN, False, 1, 0),
    ("kivi", "bfloat16", PER_CHANNEL, PER_TOKEN, False, 1, 0),
    ("rtn", "bfloat16", PER_TOKEN, PER_TOKEN, False, 1, 1),
    ("quarot", "bfloat16", PER_TOKEN, PER_TOKEN, True, 1, 1),
    ("quarot", "float16", PER_TOKEN, PER_TOKEN, True, 1, 1),
    ("vc", "float16", PER_TOKEN, PER_CHANNEL, False, 1, 1),
    ("kc_vc_mixed", "bfloat16", PER_CHANNEL, PER_CHANNEL, False, 0, 1),
]


@pytest.mark.parametrize("name,dtype,kg,vg,hadamard,kq,vq", SYM_CASES)
def test_symmetric_all_widths_bit_exact_and_attention(rq, name, dtype, kg, vg, hadamard, kq, vq):
    wl = small_wl(dtype=dtype, kg=kg, vg=vg, hadamard=hadamard, S=96, seed=61, kq=kq, vq=vq)
    bits = bits_cycle(wl.L, wl.H_kv, range(1, 9), offset=2)
    path, res, signs = run_layers(rq, wl, bits)
    for l, (k, v, q, out) in res.items():
        check_layer(path, wl, l, k, v, q, out, signs)
    assert int(path.status.item()) == 0


# ---- TurboQuant's group sizes (App. W "TurboQuant kernel"): absmax over a
# key's whole 128-channel row and over each 64-channel half of a value row;
# also min-max over the wide groups, rotated caches and per-channel partners
WIDE_CASES = [
    ("turboquant_absmax", "bfloat16", PER_TOKEN_128, PER_TOKEN_64, False, 1, 1),
    ("turboquant_absmax", "float16", PER_TOKEN_128, PER_TOKEN_64, False, 1, 1),
    ("minmax_wide", "bfloat16", PER_TOKEN_64, PER_TOKEN_128, False, 0, 0),
    ("rotated_wide", "bfloat16", PER_TOKEN_128, PER_TOKEN_64, True, 1, 1),
    ("kivi_keys_wide_values", "float16", PER_CHANNEL, PER_TOKEN_128, False, 0, 1),
]


@pytest.mark.parametrize("name,dtype,kg,vg,hadamard,kq,vq", WIDE_CASES)
def test_wide_groups_all_widths_bit_exact_and_attention(rq, name, dtype, kg, vg, hadamard, kq, vq):
    wl = small_wl(dtype=dtype, kg=kg, vg=vg, hadamard=hadamard, S=96, seed=65, kq=kq, vq=vq)
    bits = bits_cycle(wl.L, wl.H_kv, range(1, 9), offset=3)
    path, res, signs = run_layers(rq, wl, bits)
    for l, (k, v, q, out) in res.items():
        check_layer(path, wl, l, k, v, q, out, signs)
    assert int(path.status.item()) == 0


@pytest.mark.parametrize("name,dtype,kg,vg,hadamard,kq,vq", WIDE_CASES[:1] + WIDE_CASES[2:4])
def test_wide_groups_calibration_matches_oracle(rq, name, dtype, kg, vg, hadamard, kq, vq):
    wl = small_wl(L=2, H=4, S=96, dtype=dtype, hadamard=hadamard, seed=66, kg=kg, vg=vg, kq=kq, vq=vq)
    x = synth.calibration_sample(wl, T=96, device=DEV)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    mse = path.calibrate(x).cpu().numpy()
    torch.cuda.synchronize()
    n = x.shape[0]
    groupings = [wl.k_grouping if i % 2 == 0 else wl.v_grouping for i in range(n)]
    sym = [symmetric_of(wl)[i % 2] for i in range(n)]
    ref = ocalib.distortion_sweep(to_np(x), groupings, hadamard,
                                  None if signs is None else signs.numpy(), symmetric=sym)
    rel = np.abs(mse - ref) / np.abs(ref)
    assert rel.max() < MSE_RTOL, rel.max()
    assert np.all(np.diff(mse[:, 1:], axis=1) < 0)


def test_wide_groups_flag_a_non_finite_quarter(rq):
    # one NaN in a 128-channel key row makes the whole row's group bad (codes,
    # scale and zero 0, status NUMERIC), not just its quarter
    wl = small_wl(L=1, B=1, H=2, g=4, S=64, dtype="bfloat16", kg=PER_TOKEN_128, vg=PER_TOKEN_64,
                  seed=67, kq=1, vq=1)
    path = PackedKVPath(wl, DEV)
    path.set_bits(np.full((1, 2, 2), 4, dtype=np.uint8))
    k, v = synth.kv_layer(1, 2, 64, "bfloat16", 67, 0, device=DEV)
    k[0, 0, 5, 100] = float("nan")
    path.quantize(0, k, v)
    torch.cuda.synchronize()
    assert int(path.status.item()) & 1
    ol = oracle_layer(k, v, path.bits_host[0], wl.k_grouping, wl.v_grouping, False, None,
                      [(0, 0)], symmetric_of(wl))
    got = path.stream_bytes(0, 0, 0, 0).cpu().numpy()
    assert np.array_equal(got, ol[(0, 0, 0)]["words"].view(np.uint8))
    assert ol[(0, 0, 0)]["bad"][5].all()


@pytest.mark.parametrize("kq,vq", [(1, 1), (0, 1)])
def test_symmetric_tiny_values_take_the_clamped_path(rq, kq, vq):
    # |x| ~ 2^-20: scales fall in the fp16 subnormal range, codes can leave
    # 0..2M before clamping (the clamped variant of the quantizer)
    wl = small_wl(L=1, dtype="bfloat16", kg=PER_CHANNEL, vg=PER_TOKEN, S=64, seed=62,
                  kq=kq, vq=vq)
    bits = bits_cycle(1, wl.H_kv, range(1, 9), offset=1)
    path, res, signs = run_layers(rq, wl, bits, kv_scale=2.0 ** -20)
    check_layer(path, wl, 0, *res[0], signs)


@pytest.mark.parametrize("hadamard,kg,vg", [(False, PER_CHANNEL, PER_TOKEN),
                                            (True, PER_TOKEN, PER_TOKEN),
                                            (True, PER_CHANNEL, PER_CHANNEL)])
def test_symmetric_calibration_matches_oracle(rq, hadamard, kg, vg):
    wl = small_wl(L=2, H=4, S=96, dtype="bfloat16", hadamard=hadamard, seed=63, kg=kg, vg=vg,
                  kq=1, vq=0 if kg == PER_CHANNEL and not hadamard else 1)
    x = synth.calibration_sample(wl, T=96, device=DEV)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    mse = path.calibrate(x).cpu().numpy()
    torch.cuda.synchronize()
    n = x.shape[0]
    groupings = [wl.k_grouping if i % 2 == 0 else wl.v_grouping for i in range(n)]
    sym = [symmetric_of(wl)[i % 2] for i in range(n)]
    ref = ocalib.distortion_sweep(to_np(x), groupings, hadamard,
                                  None if signs is None else signs.numpy(), symmetric=sym)
    rel = np.abs(mse - ref) / np.abs(ref)
    assert rel.max() < MSE_RTOL, rel.max()
    assert np.all(np.diff(mse, axis=1) < 0)


def test_quantizer_argument_errors(rq):
    wl = small_wl(L=1, B=1, H=2, g=2, S=64, dtype="bfloat16", seed=64)
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits_cycle(1, 2, (2, 3)))
    k = torch.zeros((1, 2, 64, 128), dtype=torch.bfloat16, device=DEV)
    for kq, vq in ((2, 0), (0, -1)):
        bad = rq.make_desc(1, 1, 2, 4, 64, torch.bfloat16, 1, 0, False, kq, vq)
        with pytest.raises(rq.RQError) as e:
            rq.rq_quantize_pack(bad, 0, k, k, None, path.bits, path.offsets, path.packed)
        assert e.value.status == 1
    x = torch.zeros((2, 64, 128), dtype=torch.bfloat16, device=DEV)
    mse = torch.empty((2, 8), dtype=torch.float64, device=DEV)
    ws = torch.empty(rq.rq_calibrate_workspace_bytes(2, 64), dtype=torch.uint8, device=DEV)
    with pytest.raises(rq.RQError) as e:
        rq.rq_calibrate_distortion(x, 1, 0, False, None, mse, ws, k_quantizer=3)
    assert e.value.status == 1


