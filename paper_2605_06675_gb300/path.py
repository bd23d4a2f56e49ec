"""The whole hot path on one GPU, composed from librq calls.

calibrate (GPU sweep, b = 1..8)  ->  fit (host)  ->  allocate (host)
  ->  layout (host)  ->  quantize + pack every layer (GPU)
  ->  decode attention per layer on the packed cache (GPU)

This module only owns buffers (torch CUDA tensors) and calls the binding;
it adds no arithmetic of its own.
"""
from __future__ import annotations

import numpy as np
import torch

from . import rq
from .workloads import Workload


class PackedKVPath:
    def __init__(self, wl: Workload, device="cuda", signs: torch.Tensor | None = None):
        self.wl = wl
        self.device = torch.device(device)
        self.dtype = {"float16": torch.float16, "bfloat16": torch.bfloat16}[wl.dtype]
        self.desc = rq.make_desc(wl.L, wl.B, wl.H_kv, wl.H_q, wl.S, self.dtype, wl.k_grouping,
                                 wl.v_grouping, wl.hadamard, wl.k_quantizer, wl.v_quantizer)
        self.signs = signs.to(self.device) if (wl.hadamard and signs is not None) else None
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.bits = None
        self.offsets = None
        self.packed = None
        self.total_bytes = 0
        self._calib_ws = None
        self._mse = None
        self._dec_ws = None

    # ---- a1: distortion sweep ------------------------------------------------
    def calibrate(self, x: torch.Tensor, stream=None) -> torch.Tensor:
        """x [n][T][128] on the device -> mse [n][8] float64 on the device."""
        n, T, _ = x.shape
        need = rq.rq_calibrate_workspace_bytes(n, T)
        if self._calib_ws is None or self._calib_ws.numel() < need:
            self._calib_ws = torch.empty(need, dtype=torch.uint8, device=self.device)
        if self._mse is None or self._mse.shape[0] != n:
            self._mse = torch.empty((n, 8), dtype=torch.float64, device=self.device)
        rq.rq_calibrate_distortion(x, self.wl.k_grouping, self.wl.v_grouping, self.wl.hadamard,
                                   self.signs, self._mse, self._calib_ws, self.status, stream,
                                   self.wl.k_quantizer, self.wl.v_quantizer)
        return self._mse

    # ---- a2 + a3: fit and allocate (host) ------------------------------------
    def allocate(self, mse_host: np.ndarray, w: np.ndarray, b_lo=2, b_hi=6, r2_min=0.96):
        n = mse_host.shape[0]
        classes = np.arange(n) % 2
        alpha, beta, r2 = rq.rq_fit_distortion(mse_host, b_lo, b_hi, r2_min, classes)
        bits, obj = rq.rq_alloc(w, alpha, beta, self.wl.avg_bits, self.wl.allowed_mask)
        return bits.reshape(self.wl.L, self.wl.H_kv, 2), (alpha, beta, r2, obj)

    # ---- layout + buffers ------------------------------------------------------
    def set_bits(self, bits: np.ndarray, capacity: int | None = None):
        offsets, total = rq.rq_packed_layout(self.desc, bits)
        self.bits_host = np.asarray(bits, dtype=np.uint8).reshape(self.wl.L, self.wl.H_kv, 2)
        self.offsets_host = offsets
        # update the device tables in place when their shapes allow, so that
        # work captured in a CUDA graph reads the new widths and offsets
        bits_t = torch.from_numpy(self.bits_host.copy())
        offs_t = torch.from_numpy(offsets.view(np.int64).copy())
        if getattr(self, "bits", None) is not None and self.bits.shape == bits_t.shape:
            self.bits.copy_(bits_t)
            self.offsets.copy_(offs_t)
        else:
            self.bits = bits_t.to(self.device)
            self.offsets = offs_t.to(self.device)
        self.total_bytes = total
        cap = max(total, capacity or 0)
        if self.packed is None or self.packed.numel() < cap:
            self.packed = torch.empty(max(cap, 16), dtype=torch.uint8, device=self.device)
        return offsets, total

    # ---- a4 + a5: quantize + pack ----------------------------------------------
    def quantize(self, layer: int, k: torch.Tensor, v: torch.Tensor, stream=None):
        rq.rq_quantize_pack(self.desc, layer, k, v, self.signs, self.bits, self.offsets,
                            self.packed, self.status, stream)

    # ---- a6 + a7: decode attention -----------------------------------------------
    def decode_workspace(self) -> torch.Tensor:
        need = rq.rq_decode_workspace_bytes(self.desc)
        if self._dec_ws is None or self._dec_ws.numel() < need:
            self._dec_ws = torch.empty(max(need, 16), dtype=torch.uint8, device=self.device)
        return self._dec_ws

    def decode(self, layer: int, q: torch.Tensor, out: torch.Tensor, stream=None):
        ws = self.decode_workspace()
        rq.rq_decode_attention(self.desc, layer, q, self.packed, self.bits, self.offsets,
                               self.signs, out, ws, self.status, stream)

    # ---- decode-time append ---------------------------------------------------
    def residual(self) -> torch.Tensor:
        """The residual windows [L][B][H][2][32][128] (allocated on first use)."""
        if getattr(self, "_residual", None) is None:
            n = rq.rq_residual_bytes(self.desc)
            self._residual = torch.zeros(max(n, 16), dtype=torch.uint8, device=self.device)
        return self._residual

    def append(self, layer: int, pos: int, k_new: torch.Tensor, v_new: torch.Tensor, stream=None):
        rq.rq_append(self.desc, layer, pos, k_new, v_new, self.residual(), self.signs, self.bits,
                     self.offsets, self.packed, self.status, stream)

    def decode_len(self, layer: int, n_tokens: int, q: torch.Tensor, out: torch.Tensor,
                   stream=None):
        ws = self.decode_workspace()
        rq.rq_decode_attention_len(self.desc, layer, n_tokens, q, self.packed, self.bits,
                                   self.offsets, self.signs, self.residual(), out, ws,
                                   self.status, stream)

    def append_rows(self, layer: int, pos: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor,
                    stream=None):
        """Append one token per batch row at positions ``pos`` (CUDA int32 [B];
        negative: the row appends nothing)."""
        rq.rq_append_rows(self.desc, layer, pos, k_new, v_new, self.residual(), self.signs,
                          self.bits, self.offsets, self.packed, self.status, stream)

    def decode_rows(self, layer: int, n_tokens: torch.Tensor, q: torch.Tensor, out: torch.Tensor,
                    stream=None):
        """Decode attention, batch row b over its first n_tokens[b] tokens."""
        ws = self.decode_workspace()
        rq.rq_decode_attention_rows(self.desc, layer, n_tokens, q, self.packed, self.bits,
                                    self.offsets, self.signs, self.residual(), out, ws,
                                    self.status, stream)

    def stream_bytes(self, layer: int, batch: int, head: int, kind: int) -> torch.Tensor:
        """The packed bytes of one stream (a view into the packed buffer)."""
        off = int(self.offsets_host[layer, batch, head, kind])
        b = int(self.bits_host[layer, head, kind])
        n = (self.wl.S // 32) * 512 * (b + 1)
        return self.packed[off:off + n]
