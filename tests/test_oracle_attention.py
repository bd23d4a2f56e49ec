"""Pins for the oracle's decode attention (CPU only): special cases with a
known answer and torch's scaled_dot_product_attention as a library routine."""
import numpy as np
import pytest
import torch

from oracle import pipeline
from oracle.attention import decode_attention
from oracle.quant import PER_CHANNEL, PER_TOKEN


def test_single_token_returns_its_value():
    rng = np.random.default_rng(0)
    q = rng.standard_normal((8, 128))
    k = rng.standard_normal((2, 1, 128))
    v = rng.standard_normal((2, 1, 128))
    out = decode_attention(q, k, v)
    for j in range(8):
        assert np.allclose(out[j], v[j // 4, 0].astype(np.float32))


def test_equal_keys_average_values():
    rng = np.random.default_rng(1)
    q = rng.standard_normal((4, 128))
    k = np.repeat(rng.standard_normal((1, 1, 128)), 50, axis=1)
    v = rng.standard_normal((1, 50, 128))
    out = decode_attention(q, k, v)
    assert np.allclose(out, np.repeat(v[0].mean(axis=0, keepdims=True), 4, 0), atol=1e-6)


def test_matches_torch_sdpa():
    rng = np.random.default_rng(2)
    Hq, Hkv, S = 8, 2, 77
    q = rng.standard_normal((Hq, 128))
    k = rng.standard_normal((Hkv, S, 128))
    v = rng.standard_normal((Hkv, S, 128))
    out = decode_attention(q, k, v)
    tq = torch.tensor(q)[:, None, :]                                 # [Hq, 1, d]
    tk = torch.tensor(k).repeat_interleave(Hq // Hkv, dim=0)         # [Hq, S, d]
    tv = torch.tensor(v).repeat_interleave(Hq // Hkv, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv)[:, 0, :].numpy()
    assert np.allclose(out, ref.astype(np.float32), rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("kg", [PER_CHANNEL, PER_TOKEN])
def test_8bit_integer_cache_reduces_to_plain_attention(kg):
    # Integer data in [0, 255] with both ends in every group: at b = 8 the
    # quantizer is exact (scale 1, zero 0), so the whole pipeline equals
    # plain softmax attention on the original cache (torch SDPA, fp64).
    rng = np.random.default_rng(3)
    B, H, S = 1, 2, 64
    k = rng.integers(0, 256, size=(B, H, S, 128)).astype(np.float32)
    v = rng.integers(0, 256, size=(B, H, S, 128)).astype(np.float32)
    for x in (k, v):
        x[:, :, 0::32, :] = 0.0
        x[:, :, 1::32, :] = 255.0
        x[:, :, :, 0::32] = 0.0
        x[:, :, :, 1::32] = 255.0
    q = rng.standard_normal((B, 8, 128)).astype(np.float32) * 0.01
    bits = np.full((H, 2), 8)
    ql = pipeline.quantize_layer(k, v, bits, kg, PER_TOKEN)
    for key, r in ql.items():
        x = k if key[2] == 0 else v
        assert np.array_equal(r["xhat"], x[key[0], key[1]].astype(np.float64))
    out = pipeline.attend_layer(q, ql)
    tq = torch.tensor(q[0], dtype=torch.float64)[:, None, :]
    tk = torch.tensor(k[0], dtype=torch.float64).repeat_interleave(4, dim=0)
    tv = torch.tensor(v[0], dtype=torch.float64).repeat_interleave(4, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv)[:, 0, :].numpy()
    assert np.allclose(out[0], ref, rtol=1e-6, atol=1e-4)


def test_rotated_pipeline_close_to_plain_attention():
    # Hadamard + 8-bit: the un-rotated dequantized cache is within the
    # quantization error of the original, so attention is close to plain.
    rng = np.random.default_rng(4)
    B, H, S = 1, 1, 96
    k = rng.standard_normal((B, H, S, 128)).astype(np.float32)
    v = rng.standard_normal((B, H, S, 128)).astype(np.float32)
    signs = rng.choice([-1, 1], size=128).astype(np.int8)
    q = rng.standard_normal((B, 4, 128)).astype(np.float32)
    ql = pipeline.quantize_layer(k, v, np.full((H, 2), 8), PER_TOKEN, PER_TOKEN,
                                 hadamard=True, signs=signs)
    assert np.abs(ql[(0, 0, 0)]["xhat"] - k[0, 0]).max() < 0.02
    out = pipeline.attend_layer(q, ql)
    ref = decode_attention(q[0], k[0].astype(np.float64), v[0].astype(np.float64))
    assert np.abs(out[0] - ref).max() < 0.02


def test_residual_attention_reduces_to_its_parts():
    # with no residual token it is the packed-cache attention; with no packed
    # block it is exact attention over the raw tokens
    from oracle import pipeline as opipe
    rng = np.random.default_rng(12)
    B, H, Hq, S = 1, 2, 4, 64
    k = rng.standard_normal((B, H, S, 128)).astype(np.float32)
    v = rng.standard_normal((B, H, S, 128)).astype(np.float32)
    q = rng.standard_normal((B, Hq, 128)).astype(np.float32)
    bits = np.array([[2, 3], [4, 2]])
    ol = opipe.quantize_layer(k, v, bits, 1, 0)
    empty = np.zeros((B, H, 0, 128), np.float32)
    assert np.array_equal(opipe.attend_with_residual(q, ol, empty, empty), opipe.attend_layer(q, ol))
    got = opipe.attend_with_residual(q, {}, k[:, :, :20], v[:, :, :20])
    for h in range(H):
        for j in range(2):
            s = (k[0, h, :20].astype(np.float64) @ q[0, 2 * h + j]) / np.sqrt(128)
            p = np.exp(s - s.max())
            want = (p @ v[0, h, :20].astype(np.float64)) / p.sum()
            assert np.allclose(got[0, 2 * h + j], want, rtol=1e-6, atol=1e-6)
