"""Whole-layer oracle helpers: quantize + pack every stream, dequantize, attend.

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Composes ``quant``, ``pack`` and ``attention`` without adding arithmetic: the
cache of one layer is K, V [B][H_kv][S][128]; stream (batch, head, kind) uses
bit-width bits[head][kind] and the kind's grouping; with ``hadamard`` both K
and V are rotated per token before quantization (QuaRot reading) and the
dequantized cache is rotated back before attention.
"""
from __future__ import annotations

import numpy as np

from . import pack
from .attention import decode_attention, unrotate
from .quant import quantize_stream, storage_grouping


def quantize_layer(k, v, bits, k_grouping, v_grouping, hadamard=False, signs=None,
                   streams=None, symmetric=False):
    """Quantize and pack one layer.

    bits [H][2]. ``streams`` optionally restricts work to a list of
    (batch, head) pairs (for sampled checks at large sizes). ``symmetric``:
    the quantizer form (``quant.MINMAX`` / ``ABSMAX`` / ``LLOYDMAX``; a bool
    means min-max / absmax), one, or a (keys, values) pair.
    Returns {(batch, head, kind): dict(words=uint32[...], xhat=fp64 [S,128]
    in the original domain, bad=bool groups)}.
    """
    k = np.asarray(k, dtype=np.float32)
    v = np.asarray(v, dtype=np.float32)
    B, H, S, d = k.shape
    bits = np.asarray(bits).reshape(H, 2)
    if streams is None:
        streams = [(bb, h) for bb in range(B) for h in range(H)]
    sym = np.broadcast_to(np.asarray(symmetric, dtype=np.int64), (2,))
    out = {}
    for bb, h in streams:
        for kind, x, grouping in ((pack.KIND_K, k, k_grouping), (pack.KIND_V, v, v_grouping)):
            b = int(bits[h, kind])
            r = quantize_stream(x[bb, h], grouping, b, signs, hadamard, int(sym[kind]))
            words = pack.pack_stream(r["codes"], r["scale"], r["zero"], kind,
                                     storage_grouping(grouping), b)
            xhat = r["xhat"].astype(np.float64)
            if hadamard:
                xhat = unrotate(xhat, signs)
            out[(bb, h, kind)] = {"words": words, "xhat": xhat, "bad": r["bad"],
                                  "codes": r["codes"], "scale": r["scale"], "zero": r["zero"]}
    return out


def attend_layer(q, qlayer, batches=None, heads=None):
    """Decode attention for one layer from ``quantize_layer`` output.

    q [B][H_q][128]. Returns out [B][H_q][128] float32 (rows not requested
    stay zero). ``heads`` restricts to a list of kv heads.
    """
    q = np.asarray(q, dtype=np.float32)
    B, Hq, d = q.shape
    kv_heads = sorted({h for (_, h, _) in qlayer})
    Hkv = max(kv_heads) + 1
    g = None
    out = np.zeros((B, Hq, d), dtype=np.float32)
    batches = range(B) if batches is None else batches
    for bb in batches:
        for h in (kv_heads if heads is None else heads):
            if (bb, h, 0) not in qlayer:
                continue
            kh = qlayer[(bb, h, 0)]["xhat"][None]
            vh = qlayer[(bb, h, 1)]["xhat"][None]
            g = Hq // Hkv if g is None else g
            qs = q[bb, h * g:(h + 1) * g]
            out[bb, h * g:(h + 1) * g] = decode_attention(qs, kh, vh)
    return out


def attend_with_residual(q, qlayer, k_res, v_res, batches=None, heads=None):
    """Decode attention over a packed prefix plus unquantized residual tokens
    (decode-time append: the open 32-token block stays unquantized, as in
    KIVI's residual, Sec. 2; allocation is uniform over positions, appendix
    "Scope and Extensions").

    q [B][H_q][128]; ``qlayer``: ``quantize_layer`` output of the packed prefix
    (empty dict when no block is packed yet); k_res, v_res [B][H_kv][R][128]
    the residual tokens in the original domain (R may be 0). Returns out
    [B][H_q][128] float32.
    """
    q = np.asarray(q, dtype=np.float32)
    k_res = np.asarray(k_res, dtype=np.float64)
    v_res = np.asarray(v_res, dtype=np.float64)
    B, Hq, d = q.shape
    Hkv = k_res.shape[1]
    g = Hq // Hkv
    out = np.zeros((B, Hq, d), dtype=np.float32)
    for bb in (range(B) if batches is None else batches):
        for h in (range(Hkv) if heads is None else heads):
            kh, vh = k_res[bb, h], v_res[bb, h]
            if (bb, h, 0) in qlayer:
                kh = np.concatenate([qlayer[(bb, h, 0)]["xhat"], kh], axis=0)
                vh = np.concatenate([qlayer[(bb, h, 1)]["xhat"], vh], axis=0)
            out[bb, h * g:(h + 1) * g] = decode_attention(q[bb, h * g:(h + 1) * g], kh[None],
                                                          vh[None])
    return out
