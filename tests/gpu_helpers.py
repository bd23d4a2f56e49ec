"""Shared helpers for the GPU parity tests: run a layer through librq and the
same layer through the oracle, on identical seeded inputs."""
from __future__ import annotations

import os

import numpy as np
import torch

from oracle import pipeline as opipe

TOL = 2e-3   # attention: max |o_gpu - o_oracle| <= TOL * max(1, max |o_oracle|)


def ensure_built():
    from paper_2605_06675_gb300 import build
    srcs = [os.path.join(build.CSRC, f) for f in os.listdir(build.CSRC)]
    srcs.append(os.path.join(build.INCLUDE, "rq.h"))
    if not os.path.exists(build.LIB) or os.path.getmtime(build.LIB) < max(map(os.path.getmtime, srcs)):
        build.build()
    from paper_2605_06675_gb300 import rq
    rq.lib()
    return rq


def bits_cycle(L, H, allowed, offset=0):
    allowed = list(allowed)
    b = np.zeros((L, H, 2), dtype=np.uint8)
    for l in range(L):
        for h in range(H):
            for k in range(2):
                b[l, h, k] = allowed[(offset + l * 2 * H + 2 * h + k) % len(allowed)]
    return b


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def oracle_layer(k, v, bits_layer, kg, vg, hadamard, signs, streams=None, symmetric=False):
    """Oracle quantize+pack of the requested (batch, head) streams of one
    layer; only those slices are copied to the host."""
    sg = None if signs is None else signs.cpu().numpy()
    B, H = k.shape[0], k.shape[1]
    if streams is None:
        streams = [(bb, h) for bb in range(B) for h in range(H)]
    out = {}
    for bb, h in streams:
        kk = to_np(k[bb:bb + 1, h:h + 1])
        vv = to_np(v[bb:bb + 1, h:h + 1])
        r = opipe.quantize_layer(kk, vv, np.asarray(bits_layer)[h:h + 1], kg, vg, hadamard, sg,
                                 symmetric=symmetric)
        for kind in (0, 1):
            out[(bb, h, kind)] = r[(0, 0, kind)]
    return out


def oracle_attention(q, ol, g):
    """{(batch, q head): out[128]} for every stream pair in ``ol``."""
    from oracle.attention import decode_attention
    res = {}
    for (bb, h, kind), r in ol.items():
        if kind != 0:
            continue
        qs = to_np(q[bb, h * g:(h + 1) * g])
        o = decode_attention(qs, r["xhat"][None], ol[(bb, h, 1)]["xhat"][None])
        for j in range(g):
            res[(bb, h * g + j)] = o[j]
    return res


def attn_err(out_gpu: np.ndarray, out_ref: np.ndarray) -> float:
    scale = max(1.0, float(np.abs(out_ref).max()))
    return float(np.abs(out_gpu - out_ref).max()) / scale
