"""GPU parity on the named workloads: the tiny one end to end (calibrate ->
fit -> allocate -> quantize -> decode) and one full-size layer of each large
workload, launched exactly as bench.py launches it, checked on sampled
(batch, head) streams the oracle computes one by one."""
import numpy as np
import pytest
import torch

from oracle import alloc as oalloc
from oracle import calib as ocalib
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import (LLAMA3_8B_32K, LONG_70B_128K, PER_CHANNEL,
                                              PER_TOKEN, QWEN3_8B_8K, TINY)

from .gpu_helpers import bits_cycle, ensure_built, to_np
from .test_gpu_parity import MSE_RTOL, check_layer

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def rq():
    return ensure_built()


@pytest.mark.parametrize("kg", [PER_CHANNEL, PER_TOKEN])
def test_tiny_workload_end_to_end(rq, kg):
    wl = TINY.scaled(k_grouping=kg)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, 0, wl.value_dist, DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, 0, DEV)
    # a1: calibrate on the workload's own 1024 tokens, component (h, kind)
    x = torch.stack([t for h in range(wl.H_kv) for t in (k[0, h], v[0, h])]).contiguous()
    path = PackedKVPath(wl, DEV)
    mse = path.calibrate(x).cpu().numpy()
    n = x.shape[0]
    groupings = [wl.k_grouping if i % 2 == 0 else wl.v_grouping for i in range(n)]
    ref_mse = ocalib.distortion_sweep(to_np(x), groupings)
    assert (np.abs(mse - ref_mse) / ref_mse).max() < MSE_RTOL
    # a2 + a3: fit and allocate. On the same MSE the library and the oracle
    # agree bit for bit; the oracle's own MSE (1e-6-level differences) gives
    # an allocation of the same objective value
    w = synth.importances(n, wl.sigma_lnw, wl.seed)
    bits, (alpha, beta, r2, J) = path.allocate(mse, w)
    oa, ob, _ = ocalib.fit_distortion(mse, 2, 6, 0.96, np.arange(n) % 2)
    obits, oJ = oalloc.allocate(w, oa, ob, wl.avg_bits, wl.allowed_mask)
    assert list(bits.reshape(-1)) == obits and J == oJ
    assert int(bits.sum()) == oalloc.budget(wl.avg_bits, n) == 48
    ra, rb, _ = ocalib.fit_distortion(ref_mse, 2, 6, 0.96, np.arange(n) % 2)
    rbits, _ = oalloc.allocate(w, ra, rb, wl.avg_bits, wl.allowed_mask)
    Jr = oalloc.objective(w, ra, rb, rbits)
    Jg = oalloc.objective(w, ra, rb, list(bits.reshape(-1)))
    assert abs(Jg / Jr - 1) < 1e-4
    # a5 .. a7
    path.set_bits(bits)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    path.quantize(0, k, v)
    path.decode(0, q, out)
    torch.cuda.synchronize()
    check_layer(path, wl, 0, k, v, q, out, None)
    assert int(path.status.item()) == 0


@pytest.mark.parametrize("wl", [
    LLAMA3_8B_32K, QWEN3_8B_8K, LONG_70B_128K,
    LLAMA3_8B_32K.scaled(name="llama3_absmax_keys", k_quantizer=1),            # KIVI symmetric keys
    QWEN3_8B_8K.scaled(name="qwen3_lloydmax", k_quantizer=2, v_quantizer=2),   # TurboQuant-style
], ids=lambda w: w.name)
def test_full_size_layer_sampled(rq, wl):
    bits = bits_cycle(wl.L, wl.H_kv, wl.allowed)
    layer = wl.L - 1                      # last layer: largest stream offsets
    signs = synth.hadamard_signs(wl.seed) if wl.hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    path.set_bits(bits)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, layer, wl.value_dist, DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, layer, DEV)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    path.quantize(layer, k, v)
    path.decode(layer, q, out)
    torch.cuda.synchronize()
    streams = [(0, 0), (wl.B - 1, wl.H_kv - 1)]
    check_layer(path, wl, layer, k, v, q, out, signs, streams)
    assert int(path.status.item()) == 0
    assert torch.isfinite(out).all()
    del k, v
    torch.cuda.empty_cache()


def test_llama3_bench_path_allocator_widths(rq):
    """The bench's configuration as bench.py runs it, on one full-size layer:
    calibrate on the workload's calibration sample, fit + allocate with the
    library (bit-exact against the oracle's fit and allocation on the same
    MSE), lay out every layer at the allocator's widths in a buffer of the
    bench's capacity, quantize + decode the last layer, and compare every
    (batch 0, kv head) stream and one kv head of every other batch with the
    oracle: packed bytes bit-exact, attention within the tolerance."""
    wl = LLAMA3_8B_32K
    path = PackedKVPath(wl, DEV)
    X = synth.calibration_sample(wl, device=DEV)
    mse = path.calibrate(X).cpu().numpy()
    n = X.shape[0]
    w = synth.importances(n, wl.sigma_lnw, wl.seed)
    bits, (_, _, _, J) = path.allocate(mse, w)
    oa, ob, _ = ocalib.fit_distortion(mse, 2, 6, 0.96, np.arange(n) % 2)
    obits, oJ = oalloc.allocate(w, oa, ob, wl.avg_bits, wl.allowed_mask)
    assert list(bits.reshape(-1)) == obits and J == oJ
    assert int(bits.sum()) == oalloc.budget(wl.avg_bits, n)
    # the sweep on every 37th component against the oracle's
    idx = np.arange(0, n, 37)
    xs = to_np(X[torch.as_tensor(idx, device=X.device)])
    ref_mse = ocalib.distortion_sweep(xs, [wl.k_grouping if i % 2 == 0 else wl.v_grouping
                                           for i in idx])
    assert (np.abs(mse[idx] - ref_mse) / ref_mse).max() < MSE_RTOL
    del X
    # capacity as bench.py sizes it: every stream at the widest allowed width
    cap = wl.L * wl.B * wl.H_kv * 2 * (wl.S // 32) * 512 * (max(wl.allowed) + 1)
    path.set_bits(bits, capacity=cap)
    layer = wl.L - 1
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, layer, wl.value_dist, DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, layer, DEV)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    path.quantize(layer, k, v)
    path.decode(layer, q, out)
    torch.cuda.synchronize()
    streams = [(0, h) for h in range(wl.H_kv)] + [(bb, bb % wl.H_kv) for bb in range(1, wl.B)]
    check_layer(path, wl, layer, k, v, q, out, None, streams)
    assert int(path.status.item()) == 0
    assert torch.isfinite(out).all()
    del k, v
    torch.cuda.empty_cache()
