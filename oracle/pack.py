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

Codes image: the 32x128 code tile X[t][c] (t = token in block, c = channel) is
split among 32 "lanes"; lane = 4*gid + tig. Each lane owns 16 "fragments" of 8
codes, slots e = 0..7:

  kind K:  gid = t % 8,  tig = (c % 8) // 2,  frag = 2*(c // 16) + (t // 16),
           e = (c & 1) | ((t >> 3) & 1) << 1 | ((c >> 3) & 1) << 2
  kind V:  gid = c % 8,  tig = (t % 8) // 2,  frag = 8*(t // 16) + (c // 16),
           e = (t & 1) | ((c >> 3) & 1) << 1 | ((t >> 3) & 1) << 2

  slot position in the fragment: pos = e // 2 for even e, 4 + e // 2 for odd e
  (codes a0 a2 a4 a6 first, then a1 a3 a5 a7).

  Each lane has a bit stream of 128*b bits: the code sits, LSB first, at bits
  [8*b*frag + b*pos, +b). Lane-stream word w (bits [32w, 32w+32)) is stored at
  block word 128*(w // 4) + 4*lane + (w % 4); i.e. 16-byte piece i = w // 4 of
  lane L lives at byte 16*(32 i + L).

Meta image (128 words, one fp16 pair each, low half first):

  "pair planes" -- K per-channel and V per-token. Words 0..63 hold scale pairs,
  words 64..127 the zero pairs at the same index. A word holds the values of
  two groups g0 (low half) and g1 (high half):
    K per-channel (group = channel c):  pair (c, c+1), c even,
        index = 16*((c % 8)//2) + 2*(c // 16) + ((c // 8) % 2), half = c % 2
    V per-token (group = (t, G), G = c // 32): pair (t, t+1), t even,
        p = t // 2,  index = 16*(p % 4) + 4*(p // 4) + G,  half = t % 2

  "scale-zero words" -- K per-token and V per-channel. Word = (scale, zero)
  of one group:
    K per-token (group = (t, G)):   index = 16*(t % 8) + 4*(t // 8) + G
    V per-channel (group = c):      index = 16*(c % 8) + 2*(c // 16) + (c // 8) % 2

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


def code_positions(kind: int, b: int):
    """For every (t, c) of a block tile: lane and lane-stream bit position.

    Returns (lane[32,128], bitpos[32,128]) int64 arrays.
    """
    t = np.arange(BLOCK_TOKENS)[:, None] * np.ones((1, HEAD_DIM), dtype=np.int64)
    c = np.ones((BLOCK_TOKENS, 1), dtype=np.int64) * np.arange(HEAD_DIM)[None, :]
    if kind == KIND_K:
        gid = t % 8
        tig = (c % 8) // 2
        frag = 2 * (c // 16) + (t // 16)
        e = (c & 1) | (((t >> 3) & 1) << 1) | (((c >> 3) & 1) << 2)
    else:
        gid = c % 8
        tig = (t % 8) // 2
        frag = 8 * (t // 16) + (c // 16)
        e = (t & 1) | (((c >> 3) & 1) << 1) | (((t >> 3) & 1) << 2)
    lane = 4 * gid + tig
    pos = np.where(e % 2 == 0, e // 2, 4 + e // 2)
    bitpos = 8 * b * frag + b * pos
    return lane.astype(np.int64), bitpos.astype(np.int64)


def lane_word_to_block_word(lane: np.ndarray, w: np.ndarray) -> np.ndarray:
    return 128 * (w // 4) + 4 * lane + (w % 4)


def pack_codes_blocks(tiles: np.ndarray, kind: int, b: int) -> np.ndarray:
    """Pack code tiles [nb, 32, 128] into [nb, 128*b] uint32 words, bit by bit."""
    tiles = np.asarray(tiles).astype(np.int64)
    nb = tiles.shape[0]
    assert tiles.shape[1:] == (BLOCK_TOKENS, HEAD_DIM)
    assert nb == 0 or (tiles.min() >= 0 and tiles.max() < (1 << b))
    lane, bitpos = code_positions(kind, b)
    bits = np.zeros((nb, 32, 128 * b), dtype=np.uint8)      # lane bit streams
    for k in range(b):
        bits[:, lane, bitpos + k] = ((tiles >> k) & 1).astype(np.uint8)
    lane_words = np.zeros((nb, 32, 4 * b), dtype=np.uint64)
    for j in range(32):
        lane_words |= bits[:, :, j::32].astype(np.uint64) << np.uint64(j)
    out = np.zeros((nb, 128 * b), dtype=np.uint32)
    L = np.arange(32)[:, None] * np.ones((1, 4 * b), dtype=np.int64)
    W = np.ones((32, 1), dtype=np.int64) * np.arange(4 * b)[None, :]
    out[:, lane_word_to_block_word(L, W)] = lane_words.astype(np.uint32)
    return out


def unpack_codes_blocks(words: np.ndarray, kind: int, b: int) -> np.ndarray:
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
    lane, bitpos = code_positions(kind, b)
    tile = np.zeros((nb, BLOCK_TOKENS, HEAD_DIM), dtype=np.int64)
    for k in range(b):
        tile |= bits[:, lane, bitpos + k].astype(np.int64) << k
    return tile.astype(np.uint8)


def pack_codes_block(tile: np.ndarray, kind: int, b: int) -> np.ndarray:
    """Pack a 32x128 code tile into 128*b uint32 words (bit by bit)."""
    return pack_codes_blocks(np.asarray(tile)[None], kind, b)[0]


def unpack_codes_block(words: np.ndarray, kind: int, b: int) -> np.ndarray:
    """Inverse of ``pack_codes_block``."""
    return unpack_codes_blocks(np.asarray(words)[None], kind, b)[0]


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

    For "pairs" layouts the scale goes to ``word``, the zero to ``64 + word``,
    both in ``half``. For "sz" layouts ``half`` is None: scale low, zero high.
    """
    if kind == KIND_K and grouping == PER_CHANNEL:
        c, _ = _group_indices(kind, grouping)
        word = 16 * ((c % 8) // 2) + 2 * (c // 16) + ((c // 8) % 2)
        return word, c % 2
    if kind == KIND_V and grouping == PER_TOKEN:
        t, G = _group_indices(kind, grouping)
        p = t // 2
        word = 16 * (p % 4) + 4 * (p // 4) + G
        return word, t % 2
    if kind == KIND_K and grouping == PER_TOKEN:
        t, G = _group_indices(kind, grouping)
        return 16 * (t % 8) + 4 * (t // 8) + G, None
    c, _ = _group_indices(kind, grouping)
    return 16 * (c % 8) + 2 * (c // 16) + (c // 8) % 2, None


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
        # two groups share a word: one pass per half so no index repeats
        for h in (0, 1):
            m = half == h
            out[:, word[m]] |= s[:, m] << np.uint32(16 * h)
            out[:, 64 + word[m]] |= z[:, m] << np.uint32(16 * h)
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
        sh = (16 * half).astype(np.uint32)
        s = ((words[:, word] >> sh) & 0xFFFF).astype(np.uint16)
        z = ((words[:, 64 + word] >> sh) & 0xFFFF).astype(np.uint16)
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
        out[j0:j1, :128 * b] = pack_codes_blocks(tiles[j0:j1], kind, b)
        out[j0:j1, 128 * b:] = pack_meta_blocks(sc[j0:j1], ze[j0:j1], kind, grouping)
    return out.reshape(-1)


def unpack_stream(words: np.ndarray, S: int, kind: int, grouping: int, b: int):
    """Inverse of ``pack_stream``: (codes [S,128], scale, zero) group-shaped."""
    nblk = S // BLOCK_TOKENS
    per = 128 * (b + 1)
    words = np.asarray(words, dtype=np.uint32)
    assert words.shape == (nblk * per,)
    w = words.reshape(nblk, per)
    codes = unpack_codes_blocks(w[:, :128 * b], kind, b).reshape(S, HEAD_DIM)
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
