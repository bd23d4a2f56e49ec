"""Group-wise min-max (asymmetric) and absmax (symmetric) quantizers and the
Hadamard pre-rotation (oracle).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Paper passages followed
-----------------------
* Sec. 2 / Sec. 4.1 "Base quantizers": KIVI quantizes keys per channel and
  values per token; QuaRot rotates with a Hadamard matrix and then quantizes
  per token.
* App. W "KIVI kernel": K_hat[:, j] = Q_b(K[:, j], scale_j) (per channel),
  V_hat[t, :] = Q_b(V[t, :], scale_t) (per token).
* App. W "QuaRot kernel": X_hat = Q_b(X R) R^T with R orthogonal.

The paper gives no formula for the asymmetric min-max quantizer Q_b. The
reading used here (every step in the stated precision, in this order) is:

  for one group x[0..31] (fp16/bf16 values, exact in fp32) and b in 1..8:
    v   = fp32(x) + 0.0f              (turns -0 into +0; min/max then unique)
    mn  = min v,  mx = max v          (exact)
    L   = 2^b - 1
    s32 = fp32_rn(fp32_rn(mx - mn) / L)
    scale = fp16_rn(s32),  zero = fp16_rn(mn)        (both stored)
    sf = fp32(scale), zf = fp32(zero)
    if sf == 0: every code is 0
    else:  inv = fp32_rn(1 / sf)
           t_j = fp32_rn(v_j - zf)
           c_j = clamp(rint_half_even(t_j * inv), 0, L)   (the product t_j * inv
                 taken exactly: one rounding, to the integer, from the
                 difference to the code)
    dequantized value  x_hat_j = fp32_rn(fp32_rn(fp32(c_j) * sf) + zf)

  A group holding a non-finite value, or whose fp16 scale or zero overflows,
  is a numeric failure: codes 0, scale 0, zero 0, and the failure is reported.

Symmetric variant. The paper's one printed symmetric quantizer is the absmax
form of App. W ("TurboQuant kernel"): x_hat = round(x M / a) a / M with
a = max |x| and M = 2^(b-1) - 1 (levels q a / M, q = -M..M, zero among
them); KIVI's keys (Sec. 2, "per-channel symmetric") and QuaRot's / RTN's
per-token quantizer (Sec. 4.1; App. M, Table 16) are read as this same form over the
same groups of 32. Stored as an asymmetric group (code c = q + M, so one
decoder serves both), in the same precision steps as above:
    a   = max |v|                                  (exact)
    M   = 2^(b-1) - 1
    if M == 0 (b = 1): the only level is 0: codes 0, scale 0, zero 0
    s32 = fp32_rn(a / M),  scale = fp16_rn(s32)
    zero = fp16_rn(0 - M * sf)    (M * sf is exact in fp32: 7 + 11 bits;
                                   0 - 0 = +0, so a zero scale stores +0)
    codes as above from the stored scale and zero, clamped to 0..2M
    (code 2^b - 1 is never used)
so level c sits at fp16(c sf + zf) ~ (c - M) sf, off the exact symmetric grid
only by the fp16 rounding of zero (at most 2^-12 |zero|).

TurboQuant group sizes (App. W "TurboQuant kernel": absmax per-group
symmetric, groups of 128 elements for keys and 64 for values). Reading: the
groups run along the head dimension of one token (PER_TOKEN_128: a key's
whole 128-channel row; PER_TOKEN_64: each half of a value's row); a, M, the
stored scale and zero and the codes follow the absmax steps above over the
group's 128 or 64 values (min-max works the same way over them). In the
packed format every group of 32 channels of the token stores its wide
group's (scale, zero), so the 32-token block format is unchanged.

Rotation (QuaRot reading of "Hadamard" / "random orthogonal R"):
  y = FWHT(x * sigma) * fp32_rn(1/sqrt(128)), in fp32, butterfly stages with
  stride 1, 2, 4, ..., 64 in that order; each stage maps the pair (i, i+h),
  i with bit h clear, to (a + b, a - b). sigma is a caller-supplied +-1 vector
  (all +1 when absent). R = diag(sigma) H / sqrt(128) is orthogonal.
"""
from __future__ import annotations

import numpy as np

GROUP = 32
HEAD_DIM = 128
PER_TOKEN = 0
PER_CHANNEL = 1
PER_TOKEN_64 = 2       # groups of 64 consecutive channels of one token
PER_TOKEN_128 = 3      # the whole 128-channel row of one token
# elements per group of each grouping
GROUP_LEN = {PER_TOKEN: 32, PER_CHANNEL: 32, PER_TOKEN_64: 64, PER_TOKEN_128: 128}


def storage_grouping(grouping: int) -> int:
    """The packed format's grouping of a stream: the wide per-token groups are
    stored as per-token groups of 32 whose (scale, zero) repeat their wide
    group's (reading: TurboQuant's 128 / 64-element groups in the 32-token
    block format)."""
    return PER_CHANNEL if grouping == PER_CHANNEL else PER_TOKEN

# fp32 round-to-nearest of 1/sqrt(128) = 2^-3.5
INV_SQRT_128_F32 = np.float32(0.08838834764831845)


def canonical(v: np.ndarray) -> np.ndarray:
    """fp32 values with -0 replaced by +0 (IEEE: -0 + +0 = +0)."""
    return (np.asarray(v, dtype=np.float32) + np.float32(0.0)).astype(np.float32)


def hadamard_rotate(x: np.ndarray, signs: np.ndarray | None) -> np.ndarray:
    """Rotate the last axis (length 128) by R = diag(signs) H / sqrt(128), fp32."""
    y = np.array(x, dtype=np.float32, copy=True)
    assert y.shape[-1] == HEAD_DIM
    if signs is not None:
        y = y * np.asarray(signs, dtype=np.float32)
    lead = y.shape[:-1]
    h = 1
    while h < HEAD_DIM:
        y = y.reshape(lead + (HEAD_DIM // (2 * h), 2, h))
        a = y[..., 0, :]
        b = y[..., 1, :]
        y = np.stack([a + b, a - b], axis=-2).reshape(lead + (HEAD_DIM,))
        h *= 2
    return (y * INV_SQRT_128_F32).astype(np.float32)


def quantize_groups(v: np.ndarray, b: int, symmetric: bool = False):
    """Quantize groups along the last axis (length 32, 64 or 128) at b bits.

    Returns (codes uint8, scale float16, zero float16, bad bool), the last
    three with the group shape (last axis removed). ``symmetric``: the absmax
    form (levels q max|v| / M, q = -M..M, stored as code q + M).
    """
    assert 1 <= b <= 8
    v = canonical(v)
    assert v.shape[-1] in (32, 64, 128)
    with np.errstate(all="ignore"):
        finite = np.isfinite(v).all(axis=-1)
        vv = np.where(finite[..., None], v, np.float32(0.0))
        mn = vv.min(axis=-1)
        mx = vv.max(axis=-1)
        if symmetric:
            M = np.float32(2 ** (b - 1) - 1)
            L = np.float32(2.0 * M)                       # the largest code
            a = np.maximum(np.abs(mn), np.abs(mx)).astype(np.float32)
            s32 = (a / np.float32(max(M, 1.0))).astype(np.float32) * np.float32(M > 0)
            scale = s32.astype(np.float16)
            zero = (np.float32(0.0) - M * scale.astype(np.float32)).astype(np.float16)
        else:
            L = np.float32(2 ** b - 1)
            s32 = ((mx - mn).astype(np.float32) / L).astype(np.float32)
            scale = s32.astype(np.float16)
            zero = mn.astype(np.float16)
        bad = (~finite) | (~np.isfinite(scale)) | (~np.isfinite(zero))
        sf = scale.astype(np.float32)
        zf = zero.astype(np.float32)
        ok = (~bad) & (sf != np.float32(0.0))
        inv = (np.float32(1.0) / np.where(ok, sf, np.float32(1.0))).astype(np.float32)
        d = (vv - zf[..., None]).astype(np.float32)
        # the product of two fp32 values is exact in fp64 (48 <= 53 bits)
        t = d.astype(np.float64) * inv[..., None].astype(np.float64)
        c = np.clip(np.rint(t), 0.0, float(L))
        codes = np.where(ok[..., None], c, 0.0).astype(np.uint8)
    scale = np.where(bad, np.float16(0.0), scale).astype(np.float16)
    zero = np.where(bad, np.float16(0.0), zero).astype(np.float16)
    return codes, scale, zero, bad


def dequantize_groups(codes: np.ndarray, scale: np.ndarray, zero: np.ndarray) -> np.ndarray:
    """x_hat = fp32(c) * sf + zf as two rounded fp32 operations (no FMA)."""
    sf = np.asarray(scale, dtype=np.float16).astype(np.float32)[..., None]
    zf = np.asarray(zero, dtype=np.float16).astype(np.float32)[..., None]
    prod = (codes.astype(np.float32) * sf).astype(np.float32)
    return (prod + zf).astype(np.float32)


def to_groups(x: np.ndarray, grouping: int) -> np.ndarray:
    """View one stream x[S, 128] as its groups.

    PER_TOKEN:     groups[t, G, :]   = x[t, 32G : 32G+32]
    PER_TOKEN_64:  groups[t, G, :]   = x[t, 64G : 64G+64]
    PER_TOKEN_128: groups[t, 0, :]   = x[t, :]
    PER_CHANNEL:   groups[blk, c, :] = x[32 blk : 32 blk + 32, c]   (S % 32 == 0)
    """
    S, d = x.shape
    assert d == HEAD_DIM
    if grouping != PER_CHANNEL:
        n = GROUP_LEN[grouping]
        return x.reshape(S, HEAD_DIM // n, n)
    assert S % GROUP == 0, "per-channel groups need S % 32 == 0"
    return x.reshape(S // GROUP, GROUP, HEAD_DIM).transpose(0, 2, 1)


def from_groups(g: np.ndarray, grouping: int) -> np.ndarray:
    """Inverse of ``to_groups``: back to [S, 128]."""
    if grouping != PER_CHANNEL:
        S = g.shape[0]
        return g.reshape(S, HEAD_DIM)
    nblk = g.shape[0]
    return g.transpose(0, 2, 1).reshape(nblk * GROUP, HEAD_DIM)


MINMAX, ABSMAX, LLOYDMAX = 0, 1, 2      # group quantizer forms


def quantize_stream(x: np.ndarray, grouping: int, b: int, signs: np.ndarray | None = None,
                    hadamard: bool = False, symmetric=False):
    """Quantize one (batch, head, K/V) stream x[S, 128].

    ``symmetric`` selects the group quantizer: False / MINMAX, True / ABSMAX,
    or LLOYDMAX (the codebook quantizer of ``lloydmax``).
    Returns dict with the quantizer-domain values ``y`` [S,128] (rotated when
    ``hadamard``), ``codes`` [S,128] uint8 (element order), ``scale``/``zero``/
    ``bad`` in the shape of the stored groups of 32 (for the wide per-token
    groupings each wide group's values repeated over its groups of 32;
    ``group_scale``/``group_zero`` hold one per wide group), and ``xhat``
    [S,128] fp32 in the quantizer domain.
    """
    x = np.asarray(x, dtype=np.float32)
    y = hadamard_rotate(x, signs) if hadamard else x.astype(np.float32)
    y = canonical(y)
    g = to_groups(y, grouping)
    form = int(symmetric)
    if form == LLOYDMAX:
        assert grouping == PER_TOKEN, "Lloyd-Max groups are per-token groups of 32"
        from . import lloydmax
        codes, scale, zero, bad = lloydmax.quantize_groups(g, b)
        xhat = lloydmax.dequantize_groups(codes, scale, b)
    else:
        codes, scale, zero, bad = quantize_groups(g, b, form == ABSMAX)
        xhat = dequantize_groups(codes, scale, zero)
    rep = GROUP_LEN[grouping] // GROUP if grouping != PER_CHANNEL else 1
    return {
        "y": y,
        "codes": from_groups(codes, grouping),
        "scale": np.repeat(scale, rep, axis=-1),
        "zero": np.repeat(zero, rep, axis=-1),
        "bad": np.repeat(bad, rep, axis=-1),
        "group_scale": scale,
        "group_zero": zero,
        "xhat": from_groups(xhat, grouping),
    }
