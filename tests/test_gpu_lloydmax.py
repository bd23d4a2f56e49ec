"""The Lloyd-Max codebook quantizer (RQ_LLOYDMAX) on the GPU against the
oracle: packed codes and fp16 RMS scales bit for bit at every width, with and
without the rotation, and the distortion sweep (App. F Table 8; TurboQuant's
scalar quantizer, App. W)."""
import numpy as np
import pytest
import torch

from oracle import calib as ocalib
from oracle import quant as oquant
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle, ensure_built, oracle_layer, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda"
LM = 2


def lm_wl(dtype, hadamard, seed, value_dist="gaussian", kq=LM, vq=LM, S=96):
    return Workload(f"lm{seed}", L=1, B=2, H_kv=4, H_q=16, S=S, dtype=dtype,
                    k_grouping=PER_TOKEN, v_grouping=PER_TOKEN, hadamard=hadamard,
                    allowed=tuple(range(1, 9)), avg_bits=4.0, sigma_lnw=0.5,
                    value_dist=value_dist, seed=seed, k_quantizer=kq, v_quantizer=vq)


@pytest.mark.parametrize("dtype,hadamard,kq,vq", [
    ("bfloat16", False, LM, LM), ("float16", False, LM, LM), ("bfloat16", True, LM, LM),
    ("float16", True, LM, 0), ("bfloat16", False, 1, LM)])
def test_lloydmax_packed_bit_exact(dtype, hadamard, kq, vq):
    ensure_built()
    wl = lm_wl(dtype, hadamard, 71, kq=kq, vq=vq)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    for offset in (0, 4):
        bits = bits_cycle(1, wl.H_kv, range(1, 9), offset=offset)
        path.set_bits(bits)
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, 0, wl.value_dist, DEV)
        path.quantize(0, k, v)
        torch.cuda.synchronize()
        ol = oracle_layer(k, v, path.bits_host[0], PER_TOKEN, PER_TOKEN, hadamard, signs,
                          symmetric=(kq, vq))
        for (bb, h, kind), r in ol.items():
            got = path.stream_bytes(0, bb, h, kind).cpu().numpy()
            want = r["words"].view(np.uint8)
            assert np.array_equal(got, want), (offset, bb, h, kind, int(path.bits_host[0, h, kind]))
    assert int(path.status.item()) == 0


@pytest.mark.parametrize("hadamard", [False, True])
def test_lloydmax_calibration_matches_oracle(hadamard):
    ensure_built()
    wl = lm_wl("bfloat16", hadamard, 72).scaled(L=2)
    x = synth.calibration_sample(wl, T=96, device=DEV)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    mse = path.calibrate(x).cpu().numpy()
    torch.cuda.synchronize()
    ref = ocalib.distortion_sweep(to_np(x), [PER_TOKEN] * x.shape[0], hadamard,
                                  None if signs is None else signs.numpy(),
                                  symmetric=oquant.LLOYDMAX)
    rel = np.abs(mse - ref) / np.abs(ref)
    assert rel.max() < 1e-5, rel.max()
    assert np.all(np.diff(mse, axis=1) < 0)
    assert int(path.status.item()) == 0


def test_lloydmax_needs_per_token_groups():
    rq = ensure_built()
    k = torch.zeros((1, 2, 64, 128), dtype=torch.bfloat16, device=DEV)
    bits = torch.full((1, 2, 2), 3, dtype=torch.uint8, device=DEV)
    for kg, vg, kq, vq in ((PER_CHANNEL, PER_TOKEN, LM, 0), (PER_TOKEN, PER_CHANNEL, 0, LM)):
        desc = rq.make_desc(1, 1, 2, 4, 64, torch.bfloat16, kg, vg, False, kq, vq)
        offsets, total = rq.rq_packed_layout(desc, bits.cpu().numpy())
        off = torch.from_numpy(offsets.view(np.int64).copy()).to(DEV)
        packed = torch.empty(total, dtype=torch.uint8, device=DEV)
        with pytest.raises(rq.RQError) as e:
            rq.rq_quantize_pack(desc, 0, k, k, None, bits, off, packed)
        assert e.value.status == 1


@pytest.mark.parametrize("dtype,hadamard,kq,vq,g", [
    ("bfloat16", False, LM, LM, 4), ("float16", True, LM, LM, 4), ("bfloat16", True, LM, 0, 8),
    ("float16", False, 0, LM, 1)])
def test_lloydmax_decode_matches_oracle(dtype, hadamard, kq, vq, g):
    # codebook decode: codes looked up in the fp16 levels (keys: scaled in
    # registers; values: the levels enter the MMA with the scale in P)
    from .gpu_helpers import TOL, attn_err, oracle_attention
    ensure_built()
    wl = lm_wl(dtype, hadamard, 73, kq=kq, vq=vq, S=32 * 37).scaled(H_q=4 * g)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    bits = bits_cycle(1, wl.H_kv, range(1, 9), offset=2)
    path.set_bits(bits)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, 0, wl.value_dist, DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, 0, DEV)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    path.quantize(0, k, v)
    path.decode(0, q, out)
    torch.cuda.synchronize()
    ol = oracle_layer(k, v, path.bits_host[0], PER_TOKEN, PER_TOKEN, hadamard, signs,
                      symmetric=(kq, vq))
    for (bb, h, kind), r in ol.items():
        assert np.array_equal(path.stream_bytes(0, bb, h, kind).cpu().numpy(), r["words"].view(np.uint8))
    ref = oracle_attention(q, ol, wl.g)
    keys = sorted(ref)
    got = to_np(out)
    err = attn_err(np.stack([got[bb, j] for bb, j in keys]), np.stack([ref[key] for key in keys]))
    assert err <= TOL, err
    assert int(path.status.item()) == 0
