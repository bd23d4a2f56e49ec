"""Decode-time append on the GPU against the oracle.

Tokens are appended one at a time into the residual windows; every full
window becomes a packed block, which must equal the oracle's packing of those
32 tokens bit for bit; decode attention over the first n tokens (packed
prefix + the raw residual) must match the oracle's attention over the
dequantized prefix and the exact residual tokens (allocation is uniform over
positions, appendix "Scope and Extensions"; the open block stays unquantized
as in KIVI's residual, Sec. 2)."""
import numpy as np
import pytest
import torch

from oracle import pipeline as opipe
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import TOL, attn_err, bits_cycle, ensure_built, oracle_layer, to_np

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None

CHECKPOINTS = (1, 17, 31, 32, 33, 64, 95, 96, 100, 128, 159, 160)


@pytest.mark.gpu
@pytest.mark.parametrize("dtype,kg,vg,hadamard,allowed,kq,vq", [
    ("bfloat16", PER_CHANNEL, PER_TOKEN, False, (2, 3, 4), 0, 0),
    ("float16", PER_CHANNEL, PER_TOKEN, False, (2, 3, 4, 8), 0, 0),
    ("bfloat16", PER_TOKEN, PER_TOKEN, True, (3, 5, 6, 7), 0, 0),
    ("float16", PER_TOKEN, PER_CHANNEL, False, (1, 2, 4), 0, 0),
    ("bfloat16", PER_CHANNEL, PER_TOKEN, False, (2, 3, 4, 6), 1, 0),     # KIVI symmetric keys
    ("bfloat16", PER_TOKEN, PER_TOKEN, True, (2, 4, 5, 8), 1, 1),        # QuaRot symmetric
    ("float16", PER_TOKEN, PER_TOKEN, True, (1, 3, 4, 6), 2, 2),         # Lloyd-Max codebook
])
def test_append_then_decode_matches_oracle(dtype, kg, vg, hadamard, allowed, kq, vq):
    ensure_built()
    wl = Workload("append", L=2, B=2, H_kv=2, H_q=8, S=160, dtype=dtype, k_grouping=kg,
                  v_grouping=vg, hadamard=hadamard, allowed=allowed, avg_bits=3.0, sigma_lnw=0.5,
                  value_dist="gaussian", seed=51, k_quantizer=kq, v_quantizer=vq)
    layer = 1
    signs = synth.hadamard_signs(wl.seed).to(DEV) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    bits = bits_cycle(wl.L, wl.H_kv, allowed, offset=1)
    path.set_bits(bits)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, layer, device=DEV)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    g = wl.H_q // wl.H_kv
    for pos in range(wl.S):
        path.append(layer, pos, k[:, :, pos].contiguous(), v[:, :, pos].contiguous())
        n = pos + 1
        if n not in CHECKPOINTS:
            continue
        q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed + n, layer, DEV)
        path.decode_len(layer, n, q, out)
        torch.cuda.synchronize()
        s_pk = 32 * (n // 32)
        ol = {}
        if s_pk:
            ol = oracle_layer(k[:, :, :s_pk], v[:, :, :s_pk], bits[layer], kg, vg, hadamard, signs,
                              symmetric=(kq, vq))
            for (bb, h, kind), r in ol.items():   # the packed prefix, bit for bit
                words = r["words"].view(np.uint8)
                got = path.stream_bytes(layer, bb, h, kind)[:words.size].cpu().numpy()
                assert np.array_equal(got, words), (n, bb, h, kind)
        ref = opipe.attend_with_residual(to_np(q), ol, to_np(k[:, :, s_pk:n]),
                                         to_np(v[:, :, s_pk:n]))
        err = attn_err(to_np(out), ref)
        assert err <= TOL, (n, err)
    assert int(path.status.item()) == 0


@pytest.mark.gpu
def test_append_blocks_equal_bulk_quantization():
    # a cache built by appending equals the same cache quantized in one call
    ensure_built()
    wl = Workload("append_bulk", L=1, B=3, H_kv=4, H_q=16, S=96, dtype="bfloat16",
                  k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                  allowed=(2, 3, 4, 8), avg_bits=3.0, sigma_lnw=0.5, value_dist="student_t4",
                  seed=52)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, 0, wl.value_dist, DEV)
    bits = bits_cycle(wl.L, wl.H_kv, wl.allowed)
    a = PackedKVPath(wl, DEV)
    a.set_bits(bits)
    for pos in range(wl.S):
        a.append(0, pos, k[:, :, pos].contiguous(), v[:, :, pos].contiguous())
    b = PackedKVPath(wl, DEV)
    b.set_bits(bits)
    b.quantize(0, k, v)
    torch.cuda.synchronize()
    n = int(a.offsets_host.reshape(-1)[-1]) + (wl.S // 32) * 512 * (int(bits.reshape(-1)[-1]) + 1)
    assert torch.equal(a.packed[:n], b.packed[:n])


@pytest.mark.gpu
def test_decode_len_argument_errors():
    rq = ensure_built()
    wl = Workload("append_err", L=1, B=1, H_kv=2, H_q=4, S=64, dtype="bfloat16",
                  k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                  allowed=(2, 3, 4), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian", seed=53)
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits_cycle(1, 2, wl.allowed))
    q = torch.zeros((1, 4, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.zeros((1, 4, 128), dtype=torch.float32, device=DEV)
    ws = path.decode_workspace()
    for n in (0, 65):                                  # outside 1..S
        with pytest.raises(rq.RQError) as e:
            rq.rq_decode_attention_len(path.desc, 0, n, q, path.packed, path.bits, path.offsets,
                                       None, path.residual(), out, ws)
        assert e.value.status == 1
    with pytest.raises(rq.RQError) as e:               # residual tokens but no windows
        rq.rq_decode_attention_len(path.desc, 0, 33, q, path.packed, path.bits, path.offsets,
                                   None, None, out, ws)
    assert e.value.status == 1
    kn = torch.zeros((1, 2, 128), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(rq.RQError) as e:               # position beyond the capacity
        rq.rq_append(path.desc, 0, 64, kn, kn, path.residual(), None, path.bits, path.offsets,
                     path.packed)
    assert e.value.status == 1


# ---- a ragged decode batch: every row at its own position ---------------------
@pytest.mark.gpu
@pytest.mark.parametrize("dtype,kg,vg,hadamard,allowed,kq,vq", [
    ("bfloat16", PER_CHANNEL, PER_TOKEN, False, (2, 3, 4), 0, 0),
    ("float16", PER_TOKEN, PER_TOKEN, True, (3, 4, 5), 1, 1),
])
def test_ragged_rows_append_and_decode_match_oracle(dtype, kg, vg, hadamard, allowed, kq, vq):
    """Three rows appended one token per step until each reaches its own
    length (160, 97 and 33 tokens; a row that has stopped passes position -1),
    decoded with a token count per row: each row's packed prefix bit for bit
    and its attention against the oracle's, over its own prefix and
    residual tokens."""
    ensure_built()
    lengths = (160, 97, 33)
    wl = Workload("ragged", L=2, B=3, H_kv=2, H_q=8, S=160, dtype=dtype, k_grouping=kg,
                  v_grouping=vg, hadamard=hadamard, allowed=allowed, avg_bits=3.0, sigma_lnw=0.5,
                  value_dist="gaussian", seed=57, k_quantizer=kq, v_quantizer=vq)
    layer = 0
    signs = synth.hadamard_signs(wl.seed).to(DEV) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    bits = bits_cycle(wl.L, wl.H_kv, allowed, offset=2)
    path.set_bits(bits)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, layer, device=DEV)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    checkpoints = {1, 31, 32, 33, 50, 96, 97, 98, 130, 160}
    for step in range(wl.S):
        pos = torch.tensor([step if step < n else -1 for n in lengths], dtype=torch.int32,
                           device=DEV)
        path.append_rows(layer, pos, k[:, :, step].contiguous(), v[:, :, step].contiguous())
        if step + 1 not in checkpoints:
            continue
        n_rows = [min(step + 1, n) for n in lengths]
        q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed + step, layer, DEV)
        path.decode_rows(layer, torch.tensor(n_rows, dtype=torch.int32, device=DEV), q, out)
        torch.cuda.synchronize()
        for bb, n in enumerate(n_rows):
            s_pk = 32 * (n // 32)
            ol = {}
            if s_pk:
                ol = oracle_layer(k[bb:bb + 1, :, :s_pk], v[bb:bb + 1, :, :s_pk], bits[layer], kg, vg,
                                  hadamard, signs, symmetric=(kq, vq))
                for (_, h, kind), r in ol.items():
                    words = r["words"].view(np.uint8)
                    got = path.stream_bytes(layer, bb, h, kind)[:words.size].cpu().numpy()
                    assert np.array_equal(got, words), (step, bb, h, kind)
            ref = opipe.attend_with_residual(to_np(q[bb:bb + 1]), ol, to_np(k[bb:bb + 1, :, s_pk:n]),
                                             to_np(v[bb:bb + 1, :, s_pk:n]))
            err = attn_err(to_np(out[bb:bb + 1]), ref)
            assert err <= TOL, (step, bb, n, err)
    assert int(path.status.item()) == 0


@pytest.mark.gpu
def test_ragged_rows_out_of_range_are_reported():
    ensure_built()
    wl = Workload("ragged_err", L=1, B=2, H_kv=2, H_q=4, S=64, dtype="bfloat16",
                  k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                  allowed=(2, 3, 4), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian", seed=58)
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits_cycle(1, 2, wl.allowed))
    kn = torch.zeros((2, 2, 128), dtype=torch.bfloat16, device=DEV)
    path.append_rows(0, torch.tensor([0, 64], dtype=torch.int32, device=DEV), kn, kn)   # 64 = S
    torch.cuda.synchronize()
    assert int(path.status.item()) & 4
    path.status.zero_()
    q = torch.zeros((2, 4, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.full((2, 4, 128), 7.0, dtype=torch.float32, device=DEV)
    path.decode_rows(0, torch.tensor([1, 0], dtype=torch.int32, device=DEV), q, out)      # 0 < 1
    torch.cuda.synchronize()
    assert int(path.status.item()) & 4
    assert torch.isfinite(out).all() and (out[1] == 0).all()
