"""Seeded synthetic inputs (stand-ins for Qwen3 / Llama3 KV caches and the
WikiText-2 calibration text, which this library does not need).

Holds none of the method's arithmetic: it only draws random tensors. Both
the CUDA path and the CPU oracle consume the tensors produced here.

Recipe (per layer l of a workload with seed s):
* K ~ N(0, 1); in every kv head 4 channels (a fixed draw per (layer, head),
  the same for every token) are scaled by 10 (key outlier channels).
* V ~ N(0, 1), or Student-t with 4 degrees of freedom (z / sqrt(chi2_4 / 4))
  for the heavy-tailed long-context workload.
* q ~ N(0, 1), one decode query per (batch, query head).
* fp32 draws are rounded to the workload dtype (fp16 / bf16, RN).
* Importances w_i = exp(N(0, sigma^2)) per component (log-normal, App. R).
* Hadamard signs: a +-1 draw of length 128.
Generators are torch Philox (CUDA) or the CPU generator depending on
``device``; a given (seed, device) always yields the same tensors.
"""
from __future__ import annotations

import numpy as np
import torch

HEAD_DIM = 128
N_OUTLIERS = 4
OUTLIER_SCALE = 10.0


def _dtype(name):
    return {"float16": torch.float16, "bfloat16": torch.bfloat16}[name] if isinstance(name, str) else name


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def outlier_channels(seed: int, layer: int, H: int) -> torch.Tensor:
    """[H][4] channel indices (CPU generator, device independent)."""
    g = _gen(seed * 7919 + layer * 104729 + 17, "cpu")
    return torch.stack([torch.randperm(HEAD_DIM, generator=g)[:N_OUTLIERS] for _ in range(H)])


def kv_layer(B: int, H: int, S: int, dtype, seed: int, layer: int, value_dist="gaussian",
             device="cpu"):
    """K, V [B][H][S][128] for one layer."""
    dt = _dtype(dtype)
    g = _gen(seed * 1000003 + layer * 7 + 1, device)
    idx = outlier_channels(seed, layer, H)
    k = torch.empty((B, H, S, HEAD_DIM), dtype=dt, device=device)
    v = torch.empty((B, H, S, HEAD_DIM), dtype=dt, device=device)
    for b in range(B):
        for h in range(H):
            x = torch.randn((S, HEAD_DIM), generator=g, device=device, dtype=torch.float32)
            x[:, idx[h].to(device)] *= OUTLIER_SCALE
            k[b, h] = x.to(dt)
            y = torch.randn((S, HEAD_DIM), generator=g, device=device, dtype=torch.float32)
            if value_dist == "student_t4":
                c = torch.zeros_like(y)
                for _ in range(4):
                    z = torch.randn((S, HEAD_DIM), generator=g, device=device, dtype=torch.float32)
                    c += z * z
                y = y / torch.sqrt(c / 4.0)
            v[b, h] = y.to(dt)
    return k, v


def queries(B: int, H_q: int, dtype, seed: int, layer: int, device="cpu") -> torch.Tensor:
    g = _gen(seed * 1000003 + layer * 7 + 5, device)
    return torch.randn((B, H_q, HEAD_DIM), generator=g, device=device,
                       dtype=torch.float32).to(_dtype(dtype))


def importances(n: int, sigma: float, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed * 31 + 7)
    return np.exp(rng.normal(0.0, sigma, n))


def hadamard_signs(seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed * 13 + 3, "cpu")
    s = (torch.randint(0, 2, (HEAD_DIM,), generator=g) * 2 - 1).to(torch.int8)
    return s.to(device)


def calibration_sample(wl, T: int | None = None, device="cpu", layers=None) -> torch.Tensor:
    """x [n][T][128] with component i = (l * H + h) * 2 + kind, drawn like the
    workload's own cache (keys with outlier channels, values per value_dist)."""
    T = wl.calib_T if T is None else T
    layers = range(wl.L) if layers is None else layers
    parts = []
    for l in layers:
        k, v = kv_layer(1, wl.H_kv, T, wl.dtype, wl.seed + 100, l, wl.value_dist, device)
        for h in range(wl.H_kv):
            parts.append(k[0, h])
            parts.append(v[0, h])
    return torch.stack(parts)
