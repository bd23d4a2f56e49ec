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


LAYOUTS = [(pack.KIND_K, PER_CHANNEL), (pack.KIND_K, PER_TOKEN),
           (pack.KIND_V, PER_TOKEN), (pack.KIND_V, PER_CHANNEL)]


@pytest.mark.parametrize("kind,grouping", LAYOUTS)
@pytest.mark.parametrize("b", range(1, 9))
def test_code_positions_tile_each_lane(kind, grouping, b):
    lane, bitpos = pack.code_positions(kind, grouping, b)
    used = np.zeros((32, 128 * b), dtype=np.int64)
    for k in range(b):
        np.add.at(used, (lane, bitpos[:, :, k]), 1)
    assert (used == 1).all()          # every bit of every lane used exactly once


@pytest.mark.parametrize("kind,grouping", LAYOUTS)
@pytest.mark.parametrize("b", range(1, 9))
def test_codes_round_trip(kind, grouping, b):
    rng = np.random.default_rng(b * 7 + kind + 3 * grouping)
    tile = rng.integers(0, 1 << b, size=(32, 128))
    words = pack.pack_codes_block(tile, kind, grouping, b)
    assert words.shape == (128 * b,)
    assert np.array_equal(pack.unpack_codes_block(words, kind, grouping, b), tile)


def test_hand_words_b8_K_per_channel():
    # tile X[t][c] = (3t + 5c) mod 256, K per-channel, b = 8 (2 slots per half).
    # Lane 0 (gid 0, tig 0), unit 0, register (x, y): t = 8y, c = 2x + h;
    # slot s = x + 4y -> unit word s // 2, slot s % 2 (bits 8k, 16 + 8k).
    # unit word 0: (x0,y0) c 0,1 -> 0, 5 at slot 0; (x1,y0) c 2,3 -> 10, 15
    #   at slot 1 -> 0x0F050A00 at block word 0
    # unit word 1: (x2,y0) c 4,5 -> 20, 25; (x3,y0) c 6,7 -> 30, 35 -> 0x23191E14
    # unit word 2: (x0,y1) t 8 c 0,1 -> 24, 29; (x1,y1) c 2,3 -> 34, 39 -> 0x271D2218
    # Lane 5 (gid 1, tig 1), unit word 0: t 1, c 8,9 -> 43, 48; c 10,11 -> 53, 58
    #   -> 0x3A30352B at block word 4*5 = 20
    # Lane 0, unit 1 = lane word 8 -> block word 128*2 = 256: t 0, c 32,33 ->
    #   160, 165; c 34,35 -> 170, 175 -> 0xAFA5AAA0
    t = np.arange(32)[:, None]
    c = np.arange(128)[None, :]
    tile = (3 * t + 5 * c) % 256
    w = pack.pack_codes_block(tile, pack.KIND_K, PER_CHANNEL, 8)
    assert w[0] == 0x0F050A00
    assert w[1] == 0x23191E14
    assert w[2] == 0x271D2218
    assert w[20] == 0x3A30352B
    assert w[256] == 0xAFA5AAA0


def test_hand_words_b2_V():
    # tile X[t][c] = (t + t // 8 + c) mod 4, V (per-token), b = 2.
    # Lane 0 (gid 0, tig 0), unit 0, register (x, y): t = 8y + h, c = x;
    # slot s = x + 4y -> unit word y // 2, slot x + 4 (y % 2) at bits 2k, 16 + 2k.
    # unit word 0: half 0: y0 codes x = 0,1,2,3; y1 codes (1 + x) % 4 = 1,2,3,0
    #   -> 0x39E4; half 1: y0 (1 + x) % 4, y1 (2 + x) % 4 -> 0x4E39
    #   -> 0x4E3939E4 at block word 0
    # unit word 1: half 0: y2 (2 + x) % 4, y3 (3 + x) % 4 -> 0x934E;
    #   half 1: y2 (3 + x) % 4, y3 x % 4 -> 0xE493 -> 0xE493934E at block word 1
    t = np.arange(32)[:, None]
    c = np.arange(128)[None, :]
    tile = (t + t // 8 + c) % 4
    w = pack.pack_codes_block(tile, pack.KIND_V, PER_TOKEN, 2)
    assert w[0] == 0x4E3939E4
    assert w[1] == 0xE493934E


def test_hand_words_b3_K_per_token_with_leftover():
    # tile X[t][c] = (t // 8 + 3c) mod 8, K per-token, b = 3 (5 slots of 3
    # bits per half, bit 15 spare). Lane 0, unit 0, register (x, y): t = 8x,
    # c = 2y + h, code (x + 6y + 3h) % 8. Leftover 0 = (x0, y3): codes 2 (h 0)
    # and 5 (h 1); its bit k sits at bit 15 / 31 of unit word k.
    # unit word 0 slots (x0 y0)(x1 y0)(x2 y0)(x3 y0)(x3 y3):
    #   half 0: 0 1 2 3 5 -> 0x5688 (spare 0); half 1: 3 4 5 6 0 -> 0x0D63 | 0x8000
    #   -> 0x8D635688
    # unit word 1 slots (x0 y1)(x1 y1)(x2 y1)(x3 y1)(x1 y3):
    #   half 0: 6 7 0 1 3 -> 0x323E | 0x8000; half 1: 1 2 3 4 6 -> 0x68D1 (spare 0)
    #   -> 0x68D1B23E
    # unit word 2 slots (x0 y2)(x1 y2)(x2 y2)(x3 y2)(x2 y3):
    #   half 0: 4 5 6 7 4 -> 0x4FAC (spare 0); half 1: 7 0 1 2 7 -> 0x7447 | 0x8000
    #   -> 0xF4474FAC
    t = np.arange(32)[:, None]
    c = np.arange(128)[None, :]
    tile = (t // 8 + 3 * c) % 8
    w = pack.pack_codes_block(tile, pack.KIND_K, PER_TOKEN, 3)
    assert w[0] == 0x8D635688
    assert w[1] == 0x68D1B23E
    assert w[2] == 0xF4474FAC


def test_hand_words_b6_V_per_channel_leftovers_across_words():
    # tile X[t][c] = (7t + c) mod 64, V per-channel, b = 6 (2 slots per half,
    # spare bits 12..15). Lane 0, unit 0, register (x, y): t = 8y + h, c = x.
    # Registers psi = 4x + y < 12 fill slots (psi // 2, psi % 2); x = 3 are
    # leftovers l = y, whose 6 bits run along the 4-bit spare nibbles.
    # unit word 0: slot 0 (x0 y0) 0 / 7, slot 1 (x0 y1) 56 / 63, spare = bits
    #   0..3 of leftover 0 (x3 y0: 3 / 10): half 0 0x3E00, half 1 0xAFC7
    # unit word 1: slot 0 (x0 y2) 48 / 55, slot 1 (x0 y3) 40 / 47, spare bits
    #   12,13 = leftover 0 bits 4,5 (0 / 0), 14,15 = leftover 1 (x3 y1: 59 / 2)
    #   bits 0,1 (3 / 2): half 0 0xCA30, half 1 0x8BF7
    t = np.arange(32)[:, None]
    c = np.arange(128)[None, :]
    tile = (7 * t + c) % 64
    w = pack.pack_codes_block(tile, pack.KIND_V, PER_CHANNEL, 6)
    assert w[0] == 0xAFC73E00
    assert w[1] == 0x8BF7CA30


def _h(x):
    return int(np.float16(x).view(np.uint16))


def test_hand_meta_words():
    # K per-channel, scale_c = c, zero_c = -c - 1: for the channel pair P,
    # word 2P = zeros of (2P, 2P+1), word 2P + 1 = their scales.
    c = np.arange(128)
    w = pack.pack_meta_block(c.astype(np.float16), (-c - 1).astype(np.float16),
                             pack.KIND_K, PER_CHANNEL)
    assert w[1] == (_h(1) << 16) | _h(0)           # scales of channels (0, 1)
    assert w[3] == (_h(3) << 16) | _h(2)           # scales of channels (2, 3)
    assert w[0] == (_h(-2) << 16) | _h(-1)         # zeros of channels (0, 1)
    assert w[1] == 0x3C000000 and w[3] == 0x42004000 and w[0] == 0xC000BC00
    # V per-token, group (t, G), scale = 4t + G, zero = -(4t + G): word 4Q + G
    # = scales of tokens (2Q, 2Q+1); zeros at 64 + 32(Q>>3) + 8(Q&3) + 4(G>>1)
    # + 2((Q>>2)&1) + (G&1).
    tt = np.repeat(np.arange(32), 4)
    GG = np.tile(np.arange(4), 32)
    s = (4 * tt + GG).astype(np.float16)
    w = pack.pack_meta_block(s, -s, pack.KIND_V, PER_TOKEN)
    assert w[0] == 0x44000000                       # tokens (0,1), G 0: 0, 4
    assert w[1] == 0x45003C00                       # tokens (0,1), G 1: 1, 5
    assert w[4] == 0x4A004800                       # tokens (2,3), G 0: 8, 12
    assert w[16] == 0x50805000                      # tokens (8,9), G 0: 32, 36
    # zeros: Q = 0, G = 0 -> word 64; Q = 0, G = 1 -> 65; Q = 4 (tokens 8, 9),
    # G = 0 -> 64 + 2 = 66; Q = 1 (tokens 2, 3), G = 2 -> 64 + 8 + 4 = 76;
    # Q = 8 (tokens 16, 17), G = 3 -> 64 + 32 + 4 + 1 = 101 (zeros -67, -71)
    assert w[64] == (_h(-4) << 16) | 0x8000          # -0 and -4
    assert w[65] == (_h(-5) << 16) | _h(-1)
    assert w[66] == (_h(-36) << 16) | _h(-32)
    assert w[76] == (_h(-14) << 16) | _h(-10)
    assert w[101] == (_h(-71) << 16) | _h(-67)
    # K per-token: word = (scale, zero) of group (t, G) at 16(t%8) + 4G + t//8.
    w = pack.pack_meta_block(s, -s, pack.KIND_K, PER_TOKEN)
    assert w[0] == (0x8000 << 16)                    # t = 0, G = 0: scale 0, zero -0
    assert w[1] == (_h(-32) << 16) | _h(32)          # t = 8, G = 0
    assert w[4] == (_h(-1) << 16) | _h(1)            # t = 0, G = 1
    assert w[16] == (_h(-4) << 16) | _h(4)           # t = 1, G = 0
    assert w[17] == (_h(-36) << 16) | _h(36)         # t = 9, G = 0
    # V per-channel: word c = (scale, zero) of channel c.
    w = pack.pack_meta_block(c.astype(np.float16), (-c - 1).astype(np.float16),
                             pack.KIND_V, PER_CHANNEL)
    assert w[1] == (_h(-2) << 16) | _h(1)            # c = 1
    assert w[8] == (_h(-9) << 16) | _h(8)            # c = 8


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
        sw, zw = word
        slots = np.concatenate([2 * sw + half, 2 * zw + half])
        assert sorted(slots.tolist()) == list(range(256))


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


def test_hand_meta_words_wide_groups():
    # the wide per-token groups are stored as per-token groups of 32: a key
    # row (group of 128) with scale 2.0 (0x4000) and zero -14.0 (0xCB00)
    # gives word 16 (t mod 8) + 4 G + t / 8 = 0xCB004000 for all four G
    from oracle import pipeline, quant
    x = np.zeros((1, 1, 32, 128), dtype=np.float32)
    x[..., 3] = 14.0
    ol = pipeline.quantize_layer(x, x, np.array([[4, 4]]), quant.PER_TOKEN_128, quant.PER_TOKEN_64,
                                 symmetric=(quant.ABSMAX, quant.ABSMAX))
    words = ol[(0, 0, 0)]["words"]
    meta = words[128 * 4:]
    for t in range(32):
        for G in range(4):
            assert meta[16 * (t % 8) + 4 * G + t // 8] == 0xCB004000
    # values: halves of 64; the row's second half is all zero: scale 0, zero +0
    vm = ol[(0, 0, 1)]["words"][128 * 4:]
    s, z = pack.unpack_meta_block(vm, pack.KIND_V, PER_TOKEN)
    s = s.reshape(32, 4)
    z = z.reshape(32, 4)
    assert (s[:, :2] == 2.0).all() and (z[:, :2] == -14.0).all()
    assert (s[:, 2:] == 0.0).all() and (z[:, 2:].view(np.uint16) == 0).all()
