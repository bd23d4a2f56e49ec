"""Packed mixed-bit block format (oracle), written from its definition.

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

The paper only says that per-head bit-widths live in a static lookup table
indexed by the quantizer kernel (App. M "No runtime overhead", App. U
"Runtime Analysis") and that quantize/dequantize kernels are fused
(App. W "Kernel fusion"); how codes are stored is not given. This module
restates this library's storage format element by element, bit by bit.

Streams and blocks
------------------
A stream is one (layer, batch, kv-head, kind) with kind K or V, S tokens,
head_dim 128, bit-width b = bits[layer][head][kind]. It is S/32 blocks, block j
covering tokens [32j, 32j+32). A block is 512*(b+1) bytes: the codes image
(128*b uint32 words) followed by the meta image (128 uint32 words).

Codes image: the 32x128 code tile X[t][c] (t = token in block, c = channel)
is split among 32 lanes, lane = 4*gid + tig (gid 0..7, tig 0..3). A lane owns
4 units u = 0..3; a unit is 16 registers psi = 4*x + y (class x 0..3, member
y 0..3) and a register holds two codes, half h = 0 and h = 1:

  kind K, per-channel groups:  t = 8*y + gid,        c = 32*u + 8*tig + 2*x + h
  kind K, per-token groups:    t = 8*x + gid,        c = 32*u + 8*tig + 2*y + h
  kind V (either grouping):    t = 8*y + 2*tig + h,  c = 32*u + 4*gid + x

Each lane has a stream of 4*b words; unit u owns lane words b*u .. b*u + b-1
(unit word w = 0..b-1). With n = 16 // b code slots per 16-bit half, slot
(w, k) puts the half-h code at bits [16*h + b*k, +b) of unit word w. When
b*n < 16 the bits [16*h + b*n, 16*h + 16) of the unit's words are spare; the
half-h spare stream is those bits of unit words 0, 1, ..., b-1 in order, LSB
first, and leftover register l puts its half-h code at spare-stream bits
[b*l, b*l + b). Register psi = 4x + y goes to:

  b in {1, 2, 4, 8}:  slot s = x + 4*y, i.e. (w, k) = (s // n, s % n)
  b = 3:  x=0: (0,0) (1,0) (2,0) leftover 0;  x=1: (0,1) (1,1) (2,1) (1,4)
          x=2: (0,2) (1,2) (2,2) (2,4);       x=3: (0,3) (1,3) (2,3) (0,4)
  b = 5:  x=0: (0,0) (1,0) (2,0) (3,0);       x=1: (0,1) (1,1) (2,1) (3,1)
          x=2: (4,0) (0,2) (1,2) leftover 0;  x=3: (4,1) (2,2) (3,2) (4,2)
  b = 6:  psi < 12: (psi // 2, psi % 2); psi >= 12: leftover psi - 12
  b = 7:  psi < 14: (psi // 2, psi % 2); psi >= 14: leftover psi - 14

  (members listed y = 0, 1, 2, 3). Lane-stream word w is stored at block word
  128*(w // 4) + 4*lane + (w % 4); i.e. 16-byte piece i = w // 4 of lane L
  lives at byte 16*(32 i + L).

Meta image (128 words, one fp16 pair each, low half first):

  K per-channel (group = channel c): for the channel pair P = c // 2,
      word 2P holds the zeros of channels (2P, 2P+1), word 2P + 1 their
      scales.
  K per-token (group = (t, G), G = c // 32): word 16*(t % 8) + 4*G + t // 8
      holds (scale, zero).
  V per-token (group = (t, G)): for the token pair Q = t // 2, word 4Q + G
      holds the scales of tokens (2Q, 2Q+1), and word
      64 + 32*(Q >> 3) + 8*(Q & 3) + 4*(G >> 1) + 2*((Q >> 2) & 1) + (G & 1)
      their zeros.
  V per-channel (group = channel c): word c holds (scale, zero).

Stream order in a packed buffer (``stream_offsets``): layer, batch, kv-head,
kind (K=0, V=1); each stream starts where the previous one ends.
"""
from __future__ import annotations

import numpy as np

from .quant import GROUP, HEAD_DIM, PER_CHANNEL, PER_TOKEN

KIND_K = 0
KIND_V = 1
BLOCK_TOKENS = 32
META_WORDS = 128


def block_bytes(b: int) -> int:
    return 512 * (b + 1)


# Register psi = 4x + y of a unit -> ("slot", unit word, slot) or ("left", l).
def register_location(b: int, x: int, y: int):
    n = 16 // b
    if b in (1, 2, 4, 8):
        s = x + 4 * y
        return ("slot", s // n, s % n)
    if b == 3:
        table = {0: [(0, 0), (1, 0), (2, 0), None], 1: [(0, 1), (1, 1), (2, 1), (1, 4)],
                 2: [(0, 2), (1, 2), (2, 2), (2, 4)], 3: [(0, 3), (1, 3), (2, 3), (0, 4)]}
        loc = table[x][y]
        return ("left", 0) if loc is None else ("slot",) + loc
    if b == 5:
        table = {0: [(0, 0), (1, 0), (2, 0), (3, 0)], 1: [(0, 1), (1, 1), (2, 1), (3, 1)],
                 2: [(4, 0), (0, 2), (1, 2), None], 3: [(4, 1), (2, 2), (3, 2), (4, 2)]}
        loc = table[x][y]
        return ("left", 0) if loc is None else ("slot",) + loc
    psi = 4 * x + y
    main = 12 if b == 6 else 14
    if psi < main:
        return ("slot", psi // 2, psi % 2)
    return ("left", psi - main)


def register_element(kind: int, grouping: int, gid: int, tig: int, u: int, x: int, y: int,
                     h: int):
    """(token, channel) of half h of register (x, y) of unit u of lane (gid, tig)."""
    if kind == KIND_K and grouping == PER_CHANNEL:
        return 8 * y + gid, 32 * u + 8 * tig + 2 * x + h
    if kind == KIND_K:
        return 8 * x + gid, 32 * u + 8 * tig + 2 * y + h
    return 8 * y + 2 * tig + h, 32 * u + 4 * gid + x


def code_bit_positions(b: int, u: int, x: int, y: int, h: int):
    """Lane-stream bit positions of code bits 0..b-1 of half h of register (x, y)."""
    n = 16 // b
    spare = 16 - b * n
    loc = register_location(b, x, y)
    out = []
    for k in range(b):
        if loc[0] == "slot":
            w, slot = loc[1], loc[2]
            bit = 16 * h + b * slot + k
        else:
            i = b * loc[1] + k                     # spare-stream bit index
            w = i // spare
            bit = 16 * h + b * n + i % spare
        out.append(32 * (b * u + w) + bit)
    return out


_POS_CACHE = {}


def code_positions(kind: int, grouping: int, b: int):
    """For every (t, c) of a block tile: its lane and the lane-stream bit
    positions of its code bits 0..b-1.

    Returns (lane[32,128], bitpos[32,128,b]) int64 arrays.
    """
    key = (kind, grouping, b)
    if key in _POS_CACHE:
        return _POS_CACHE[key]
    lane = np.full((BLOCK_TOKENS, HEAD_DIM), -1, dtype=np.int64)
    bitpos = np.full((BLOCK_TOKENS, HEAD_DIM, b), -1, dtype=np.int64)
    for gid in range(8):
        for tig in range(4):
            for u in range(4):
                for x in range(4):
                    for y in range(4):
                        for h in range(2):
                            t, c = register_element(kind, grouping, gid, tig, u, x, y, h)
                            assert lane[t, c] == -1
                            lane[t, c] = 4 * gid + tig
                            bitpos[t, c] = code_bit_positions(b, u, x, y, h)
    assert (lane >= 0).all()
    _POS_CACHE[key] = (lane, bitpos)
    return lane, bitpos


def lane_word_to_block_word(lane: np.ndarray, w: np.ndarray) -> np.ndarray:
    return 128 * (w // 4) + 4 * lane + (w % 4)


def pack_codes_blocks(tiles: np.ndarray, kind: int, grouping: int, b: int) -> np.ndarray:
    """Pack code tiles [nb, 32, 128] into [nb, 128*b] uint32 words, bit by bit."""
    tiles = np.asarray(tiles).astype(np.int64)
    nb = tiles.shape[0]
    assert tiles.shape[1:] == (BLOCK_TOKENS, HEAD_DIM)
    assert nb == 0 or (tiles.min() >= 0 and tiles.max() < (1 << b))
    lane, bitpos = code_positions(kind, grouping, b)
    bits = np.zeros((nb, 32, 128 * b), dtype=np.uint8)      # lane bit streams
    for k in range(b):
        bits[:, lane, bitpos[:, :, k]] = ((tiles >> k) & 1).astype(np.uint8)
    lane_words = np.zeros((nb, 32, 4 * b), dtype=np.uint64)
    for j in range(32):
        lane_words |= bits[:, :, j::32].astype(np.uint64) << np.uint64(j)
    out = np.zeros((nb, 128 * b), dtype=np.uint32)
    L = np.arange(32)[:, None] * np.ones((1, 4 * b), dtype=np.int64)
    W = np.ones((32, 1), dtype=np.int64) * np.arange(4 * b)[None, :]
    out[:, lane_word_to_block_word(L, W)] = lane_words.astype(np.uint32)
    return out


def unpack_codes_blocks(words: np.ndarray, kind: int, grouping: int, b: int) -> np.ndarray:
    """Inverse of ``pack_codes_blocks``: [nb, 128*b] words -> [nb, 32, 128] codes."""
    words = np.asarray(words, dtype=np.uint32)
    nb = words.shape[0]
    assert words.shape[1:] == (128 * b,)
    L = np.arange(32)[:, None] * np.ones((1, 4 * b), dtype=np.int64)
    W = np.ones((32, 1), dtype=np.int64) * np.arange(4 * b)[None, :]
    lane_words = words[:, lane_word_to_block_word(L, W)].astype(np.uint64)
    bits = np.zeros((nb, 32, 128 * b), dtype=np.uint8)
    for j in range(32):
        bits[:, :, j::32] = ((lane_words >> np.uint64(j)) & np.uint64(1)).astype(np.uint8)
    lane, bitpos = code_positions(kind, grouping, b)
    tile = np.zeros((nb, BLOCK_TOKENS, HEAD_DIM), dtype=np.int64)
    for k in range(b):
        tile |= bits[:, lane, bitpos[:, :, k]].astype(np.int64) << k
    return tile.astype(np.uint8)


def pack_codes_block(tile: np.ndarray, kind: int, grouping: int, b: int) -> np.ndarray:
    """Pack a 32x128 code tile into 128*b uint32 words (bit by bit)."""
    return pack_codes_blocks(np.asarray(tile)[None], kind, grouping, b)[0]


def unpack_codes_block(words: np.ndarray, kind: int, grouping: int, b: int) -> np.ndarray:
    """Inverse of ``pack_codes_block``."""
    return unpack_codes_blocks(np.asarray(words)[None], kind, grouping, b)[0]


def meta_layout(kind: int, grouping: int) -> str:
    if (kind == KIND_K and grouping == PER_CHANNEL) or (kind == KIND_V and grouping == PER_TOKEN):
        return "pairs"
    return "sz"


def _group_indices(kind: int, grouping: int):
    """Group coordinates of one block, in ``to_groups`` order.

    PER_TOKEN: groups (t, G) for t in 0..31, G in 0..3 -> arrays t, G.
    PER_CHANNEL: groups c in 0..127 -> array c.
    """
    if grouping == PER_TOKEN:
        t = np.repeat(np.arange(BLOCK_TOKENS), 4)
        G = np.tile(np.arange(4), BLOCK_TOKENS)
        return t, G
    return np.arange(HEAD_DIM), None


def meta_positions(kind: int, grouping: int):
    """For every group of a block (``to_groups`` order): (word index, half).

    For "pairs" layouts ``word`` is a pair (scale word, zero word) and both
    values go to ``half``. For "sz" layouts ``half`` is None: scale low, zero
    high in the one word.
    """
    if kind == KIND_K and grouping == PER_CHANNEL:
        c, _ = _group_indices(kind, grouping)
        P = c // 2
        return (2 * P + 1, 2 * P), c % 2
    if kind == KIND_V and grouping == PER_TOKEN:
        t, G = _group_indices(kind, grouping)
        Q = t // 2
        zw = 64 + 32 * (Q >> 3) + 8 * (Q & 3) + 4 * (G >> 1) + 2 * ((Q >> 2) & 1) + (G & 1)
        return (4 * Q + G, zw), t % 2
    if kind == KIND_K and grouping == PER_TOKEN:
        t, G = _group_indices(kind, grouping)
        return 16 * (t % 8) + 4 * G + t // 8, None
    c, _ = _group_indices(kind, grouping)
    return c, None


def pack_meta_blocks(scale: np.ndarray, zero: np.ndarray, kind: int, grouping: int) -> np.ndarray:
    """Pack per-block group (scale, zero) fp16 values [nb, 128] into [nb, 128] words."""
    s = np.asarray(scale, dtype=np.float16).reshape(-1, 128).view(np.uint16).astype(np.uint32)
    z = np.asarray(zero, dtype=np.float16).reshape(-1, 128).view(np.uint16).astype(np.uint32)
    nb = s.shape[0]
    word, half = meta_positions(kind, grouping)
    out = np.zeros((nb, META_WORDS), dtype=np.uint32)
    if half is None:
        out[:, word] = s | (z << np.uint32(16))
    else:
        sw, zw = word
        # two groups share a word: one pass per half so no index repeats
        for h in (0, 1):
            m = half == h
            out[:, sw[m]] |= s[:, m] << np.uint32(16 * h)
            out[:, zw[m]] |= z[:, m] << np.uint32(16 * h)
    return out


def pack_meta_block(scale: np.ndarray, zero: np.ndarray, kind: int, grouping: int) -> np.ndarray:
    """Pack one block's 128 group (scale, zero) fp16 values into 128 words."""
    return pack_meta_blocks(np.asarray(scale)[None], np.asarray(zero)[None], kind, grouping)[0]


def unpack_meta_blocks(words: np.ndarray, kind: int, grouping: int):
    words = np.asarray(words, dtype=np.uint32)
    word, half = meta_positions(kind, grouping)
    if half is None:
        s = (words[:, word] & 0xFFFF).astype(np.uint16)
        z = (words[:, word] >> 16).astype(np.uint16)
    else:
        sw, zw = word
        sh = (16 * half).astype(np.uint32)
        s = ((words[:, sw] >> sh) & 0xFFFF).astype(np.uint16)
        z = ((words[:, zw] >> sh) & 0xFFFF).astype(np.uint16)
    return s.view(np.float16), z.view(np.float16)


def unpack_meta_block(words: np.ndarray, kind: int, grouping: int):
    s, z = unpack_meta_blocks(np.asarray(words)[None], kind, grouping)
    return s[0], z[0]


def pack_stream(codes: np.ndarray, scale: np.ndarray, zero: np.ndarray, kind: int,
                grouping: int, b: int, chunk: int = 256) -> np.ndarray:
    """Pack one stream: codes [S,128] (element order) and group-shaped
    scale/zero (as returned by ``quant.quantize_stream``) into uint32 words:
    block j = codes image of tokens [32j, 32j+32) then its meta image."""
    S = codes.shape[0]
    assert S % BLOCK_TOKENS == 0
    nblk = S // BLOCK_TOKENS
    tiles = np.asarray(codes).reshape(nblk, BLOCK_TOKENS, HEAD_DIM)
    sc = np.asarray(scale).reshape(nblk, 128)
    ze = np.asarray(zero).reshape(nblk, 128)
    out = np.zeros((nblk, 128 * (b + 1)), dtype=np.uint32)
    for j0 in range(0, nblk, chunk):
        j1 = min(nblk, j0 + chunk)
        out[j0:j1, :128 * b] = pack_codes_blocks(tiles[j0:j1], kind, grouping, b)
        out[j0:j1, 128 * b:] = pack_meta_blocks(sc[j0:j1], ze[j0:j1], kind, grouping)
    return out.reshape(-1)


def unpack_stream(words: np.ndarray, S: int, kind: int, grouping: int, b: int):
    """Inverse of ``pack_stream``: (codes [S,128], scale, zero) group-shaped."""
    nblk = S // BLOCK_TOKENS
    per = 128 * (b + 1)
    words = np.asarray(words, dtype=np.uint32)
    assert words.shape == (nblk * per,)
    w = words.reshape(nblk, per)
    codes = unpack_codes_blocks(w[:, :128 * b], kind, grouping, b).reshape(S, HEAD_DIM)
    s, z = unpack_meta_blocks(w[:, 128 * b:], kind, grouping)
    if grouping == PER_TOKEN:
        return codes, s.reshape(S, 4), z.reshape(S, 4)
    return codes, s.reshape(nblk, HEAD_DIM), z.reshape(nblk, HEAD_DIM)


def stream_offsets(L: int, B: int, H: int, S: int, bits: np.ndarray) -> tuple[np.ndarray, int]:
    """Byte offset of every stream [L][B][H][2] and the total buffer size."""
    bits = np.asarray(bits).reshape(L, H, 2)
    nblk = S // BLOCK_TOKENS
    off = np.zeros((L, B, H, 2), dtype=np.uint64)
    pos = 0
    for l in range(L):
        for bb in range(B):
            for h in range(H):
                for kind in range(2):
                    off[l, bb, h, kind] = pos
                    pos += nblk * block_bytes(int(bits[l, h, kind]))
    return off, pos
