"""Pins for the oracle's packed block format (CPU only).

The format is this library's own (the paper stores codes in an unspecified
way behind a per-head lookup table, App. M / App. U). The pins: every code
lands on its own bit range and the ranges tile each lane exactly; pack and
unpack round-trip; a handful of words derived by hand from the format text
(the derivations are in the comments); the codes-only byte count equals the
paper's Table 12.
"""
import os

import numpy as np
import pytest

from oracle import pack
from oracle.quant import PER_CHANNEL, PER_TOKEN

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.mark.parametrize("kind", [pack.KIND_K, pack.KIND_V])
@pytest.mark.parametrize("b", range(1, 9))
def test_code_positions_tile_each_lane(kind, b):
    lane, bitpos = pack.code_positions(kind, b)
    used = np.zeros((32, 128 * b), dtype=np.int64)
    for k in range(b):
        np.add.at(used, (lane, bitpos + k), 1)
    assert (used == 1).all()          # every bit of every lane used exactly once


@pytest.mark.parametrize("kind", [pack.KIND_K, pack.KIND_V])
@pytest.mark.parametrize("b", range(1, 9))
def test_codes_round_trip(kind, b):
    rng = np.random.default_rng(b * 7 + kind)
    tile = rng.integers(0, 1 << b, size=(32, 128))
    words = pack.pack_codes_block(tile, kind, b)
    assert words.shape == (128 * b,)
    assert np.array_equal(pack.unpack_codes_block(words, kind, b), tile)


def test_hand_words_b8_K():
    # tile X[t][c] = (3t + 5c) mod 256, kind K, b = 8.
    # Lane 0 (gid 0, tig 0), fragment 0 (c < 16, t < 16) holds t in {0, 8},
    # c in {0, 1, 8, 9}; slots: pos0 (0,0) pos1 (8,0) pos2 (0,8) pos3 (8,8)
    # pos4 (0,1) pos5 (8,1) pos6 (0,9) pos7 (8,9); one byte each.
    # lane word 0 = [0, 24, 40, 64] -> 0x40281800 at block word 0
    # lane word 1 = [5, 29, 45, 69] -> 0x452D1D05 at block word 1
    # Lane 5 (gid 1, tig 1), word 0: (1,2) (9,2) (1,10) (9,10) = 13 37 53 77
    #   -> 0x4D35250D at block word 4*5 = 20
    # Lane 0, word 4 = fragment 2 (16 <= c < 32) low half:
    #   (0,16) (8,16) (0,24) (8,24) = 80 104 120 144 -> 0x90786850 at word 128
    t = np.arange(32)[:, None]
    c = np.arange(128)[None, :]
    tile = (3 * t + 5 * c) % 256
    w = pack.pack_codes_block(tile, pack.KIND_K, 8)
    assert w[0] == 0x40281800
    assert w[1] == 0x452D1D05
    assert w[20] == 0x4D35250D
    assert w[128] == 0x90786850


def test_hand_words_b2_V():
    # tile X[t][c] = (t + c // 8) mod 4, kind V, b = 2.
    # Lane 0 (gid 0, tig 0): channels c % 8 == 0, tokens t % 8 in {0, 1}.
    # Fragment 0 (t < 16, c < 16): pos0 (0,0)=0 pos1 (0,8)=1 pos2 (8,0)=0
    #   pos3 (8,8)=1 pos4 (1,0)=1 pos5 (1,8)=2 pos6 (9,0)=1 pos7 (9,8)=2
    #   -> 2-bit fields -> 0x9944
    # Fragment 1 (16 <= c < 32): pos0 (0,16)=2 pos1 (0,24)=3 pos2 (8,16)=2
    #   pos3 (8,24)=3 pos4 (1,16)=3 pos5 (1,24)=0 pos6 (9,16)=3 pos7 (9,24)=0
    #   -> 0x33EE
    # lane word 0 = 0x9944 | 0x33EE << 16 = 0x33EE9944 at block word 0
    t = np.arange(32)[:, None]
    c = np.arange(128)[None, :]
    tile = (t + c // 8) % 4
    w = pack.pack_codes_block(tile, pack.KIND_V, 2)
    assert w[0] == 0x33EE9944


def _h(x):
    return int(np.float16(x).view(np.uint16))


def test_hand_meta_words():
    # K per-channel, scale_c = c, zero_c = -c - 1 ("pair planes").
    c = np.arange(128)
    w = pack.pack_meta_block(c.astype(np.float16), (-c - 1).astype(np.float16),
                             pack.KIND_K, PER_CHANNEL)
    assert w[0] == (_h(1) << 16) | _h(0)           # channels (0, 1)
    assert w[1] == (_h(9) << 16) | _h(8)           # channels (8, 9)
    assert w[16] == (_h(3) << 16) | _h(2)          # channels (2, 3)
    assert w[64] == (_h(-2) << 16) | _h(-1)        # zeros of channels (0, 1)
    assert w[0] == 0x3C000000 and w[1] == 0x48804800 and w[64] == 0xC000BC00
    # V per-token, group (t, G), scale = 4t + G ("pair planes").
    tt = np.repeat(np.arange(32), 4)
    GG = np.tile(np.arange(4), 32)
    s = (4 * tt + GG).astype(np.float16)
    w = pack.pack_meta_block(s, np.zeros(128, np.float16), pack.KIND_V, PER_TOKEN)
    assert w[0] == 0x44000000                       # tokens (0,1), G 0: 0, 4
    assert w[1] == 0x45003C00                       # tokens (0,1), G 1: 1, 5
    assert w[4] == 0x50805000                       # tokens (8,9), G 0: 32, 36
    assert w[16] == 0x4A004800                      # tokens (2,3), G 0: 8, 12
    # K per-token: word = (scale, zero) of group (t, G) at 16(t%8) + 4(t//8) + G.
    w = pack.pack_meta_block(s, -s, pack.KIND_K, PER_TOKEN)
    assert w[0] == (0x8000 << 16)                    # t = 0, G = 0: scale 0, zero -0
    assert w[4] == (_h(-32) << 16) | _h(32)          # t = 8, G = 0
    assert w[16] == (_h(-4) << 16) | _h(4)           # t = 1, G = 0
    assert w[17] == (_h(-5) << 16) | _h(5)           # t = 1, G = 1
    # V per-channel: word 16(c%8) + 2(c//16) + (c//8)%2.
    w = pack.pack_meta_block(c.astype(np.float16), (-c - 1).astype(np.float16),
                             pack.KIND_V, PER_CHANNEL)
    assert w[1] == (_h(-9) << 16) | _h(8)            # c = 8
    assert w[2] == (_h(-17) << 16) | _h(16)          # c = 16
    assert w[16] == (_h(-2) << 16) | _h(1)           # c = 1


@pytest.mark.parametrize("kind,grouping", [(0, PER_CHANNEL), (0, PER_TOKEN),
                                           (1, PER_TOKEN), (1, PER_CHANNEL)])
def test_meta_round_trip(kind, grouping):
    rng = np.random.default_rng(kind * 3 + grouping)
    s = rng.standard_normal(128).astype(np.float16)
    z = rng.standard_normal(128).astype(np.float16)
    w = pack.pack_meta_block(s, z, kind, grouping)
    s2, z2 = pack.unpack_meta_block(w, kind, grouping)
    assert np.array_equal(s2.view(np.uint16), s.view(np.uint16))
    assert np.array_equal(z2.view(np.uint16), z.view(np.uint16))
    word, half = pack.meta_positions(kind, grouping)
    if half is None:
        assert sorted(word.tolist()) == list(range(128))
    else:
        assert sorted((2 * word + half).tolist()) == list(range(128))


def test_stream_round_trip():
    from oracle.quant import quantize_stream
    rng = np.random.default_rng(4)
    x = rng.standard_normal((96, 128)).astype(np.float32)
    for kind, grouping in ((0, PER_CHANNEL), (1, PER_TOKEN), (0, PER_TOKEN), (1, PER_CHANNEL)):
        for b in (1, 3, 8):
            r = quantize_stream(x, grouping, b)
            words = pack.pack_stream(r["codes"], r["scale"], r["zero"], kind, grouping, b)
            assert words.size * 4 == 3 * pack.block_bytes(b)
            codes, sc, ze = pack.unpack_stream(words, 96, kind, grouping, b)
            assert np.array_equal(codes, r["codes"])
            assert np.array_equal(sc.view(np.uint16), r["scale"].view(np.uint16))
            assert np.array_equal(ze.view(np.uint16), r["zero"].view(np.uint16))


def test_table12_codes_only_bytes():
    # Codes bytes of a cache = sum over streams of (S/32) * 512 * b. With the
    # paper's bits-only accounting this must give Table 12 at seq 4096:
    # uniform 4 bits and half the heads at 3 / half at 4 (average 3.5).
    rows = [l.split() for l in open(os.path.join(GOLDEN, "table12_memory.txt"))
            if l.strip() and not l.startswith("#")]
    MiB = 1024 * 1024
    for name, L, H, fp16_mb, b4_mb, b35_mb in rows:
        L, H = int(L), int(H)
        S = 4096
        nblk = S // 32
        fp16 = L * H * 2 * S * 128 * 2
        assert fp16 == int(fp16_mb) * MiB
        bits4 = np.full((L, H, 2), 4)
        bits35 = np.full((L, H, 2), 4)
        bits35[:, : H // 2, :] = 3
        for bits, want in ((bits4, b4_mb), (bits35, b35_mb)):
            off, total = pack.stream_offsets(L, 1, H, S, bits)
            codes_only = int(sum(nblk * 512 * int(b) for b in bits.reshape(-1)))
            meta = L * H * 2 * nblk * 512
            assert total == codes_only + meta
            assert codes_only == int(want) * MiB


def test_stream_offsets_order():
    bits = np.array([[[2, 3], [4, 8]]])     # L=1, H=2
    off, total = pack.stream_offsets(1, 2, 2, 64, bits)
    nb = 2
    sizes = [nb * pack.block_bytes(b) for b in (2, 3, 4, 8)]
    expect = np.cumsum([0] + sizes * 2)[:-1].reshape(1, 2, 2, 2)
    assert np.array_equal(off.astype(np.int64), expect)
    assert total == 2 * sum(sizes)
