"""Decode attention on the dequantized mixed-bit cache (oracle), fp64.

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.

Paper passages followed
-----------------------
* Sec. 1: each new token attends to all cached key/value pairs (decode).
* Sec. 4.1 "Models": GQA, head_dim 128; query head j reads kv head j // g,
  g = H_q / H_kv.
* App. W "QuaRot kernel": X_hat = Q_b(X R) R^T -- the rotated cache is
  rotated back before use. This oracle un-rotates the dequantized K and V
  explicitly (K_hat = K_hat' R^T) and runs plain attention in the original
  domain, which is a different formulation from rotating q.

Reading: softmax scale 1/sqrt(128); no mask (one decode query attends every
cached token); scores, softmax and the weighted sum in fp64; the result is
cast to fp32 at the end.
"""
from __future__ import annotations

import numpy as np

from .quant import HEAD_DIM


def sylvester_hadamard(n: int = HEAD_DIM) -> np.ndarray:
    """Unnormalised Sylvester Hadamard matrix H_n (entries +-1), fp64."""
    H = np.ones((1, 1))
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    return H


def rotation_matrix(signs=None, n: int = HEAD_DIM) -> np.ndarray:
    """R = diag(signs) H / sqrt(n), so that a row x maps to x R."""
    s = np.ones(n) if signs is None else np.asarray(signs, dtype=np.float64)
    return (s[:, None] * sylvester_hadamard(n)) / np.sqrt(n)


def unrotate(xhat_rot: np.ndarray, signs=None) -> np.ndarray:
    """x_hat = x_hat' R^T (fp64)."""
    R = rotation_matrix(signs, xhat_rot.shape[-1])
    return np.asarray(xhat_rot, dtype=np.float64) @ R.T


def decode_attention(q: np.ndarray, k_hat: np.ndarray, v_hat: np.ndarray) -> np.ndarray:
    """q [H_q, d]; k_hat, v_hat [H_kv, S, d] (dequantized, original domain).

    Returns out [H_q, d] float32.
    """
    q = np.asarray(q, dtype=np.float64)
    k_hat = np.asarray(k_hat, dtype=np.float64)
    v_hat = np.asarray(v_hat, dtype=np.float64)
    Hq, d = q.shape
    Hkv = k_hat.shape[0]
    g = Hq // Hkv
    out = np.zeros((Hq, d), dtype=np.float64)
    scale = 1.0 / np.sqrt(d)
    for j in range(Hq):
        h = j // g
        s = (k_hat[h] @ q[j]) * scale
        m = np.max(s)
        p = np.exp(s - m)
        out[j] = (p @ v_hat[h]) / np.sum(p)
    return out.astype(np.float32)
