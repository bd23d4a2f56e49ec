"""Thin Python binding of librq (``include/rq.h``): same names, argument
marshalling only. Every step of the path runs in librq's kernels/host code.

Host arrays are numpy; device buffers are torch CUDA tensors (PyTorch is used
for device memory and streams only). Errors raise ``RQError``. There is no
fallback: if librq.so is missing the first call raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "librq.so")

RQ_OK = 0
RQ_F16, RQ_BF16 = 0, 1
RQ_PER_TOKEN, RQ_PER_CHANNEL, RQ_PER_TOKEN_64, RQ_PER_TOKEN_128 = 0, 1, 2, 3
RQ_MINMAX, RQ_ABSMAX, RQ_LLOYDMAX = 0, 1, 2
RQ_CAP_5X = 1
RQ_STATUS_NUMERIC = 1
RQ_STATUS_BAD_BITS = 2
RQ_STATUS_BAD_POSITION = 4
RQ_DECODE_BACK_TO_BACK = 0      # rq_decode_pattern
RQ_DECODE_INTERLEAVED = 1
RQ_STATIC_SCRATCH_BYTES = 8 << 20
HEAD_DIM = 128
GROUP = 32

STATUS_NAMES = {0: "RQ_OK", 1: "RQ_ERR_INVALID_ARG", 2: "RQ_ERR_INFEASIBLE", 3: "RQ_ERR_SHAPE",
                4: "RQ_ERR_ALIGNMENT", 5: "RQ_ERR_WORKSPACE", 6: "RQ_ERR_CUDA"}

# every symbol include/rq.h declares
EXPORTS = ["rq_status_string", "rq_abi_version", "rq_lloydmax_levels", "rq_fit_distortion", "rq_alloc",
           "rq_alloc_continuous", "rq_packed_layout", "rq_calibrate_workspace_bytes",
           "rq_calibrate_distortion", "rq_quantize_pack", "rq_decode_workspace_bytes",
           "rq_decode_attention", "rq_decode_attention_static", "rq_residual_bytes",
           "rq_append", "rq_decode_attention_len", "rq_append_rows", "rq_decode_attention_rows",
           "rq_decode_set_pattern"]


class RQError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)}")


class rq_cache_desc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("L", "B", "H_kv", "H_q", "S", "d", "group", "dtype", "k_grouping",
                 "v_grouping", "hadamard", "k_quantizer", "v_quantizer")]


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int32
_U = ctypes.c_uint32
_D = ctypes.c_double
_SZ = ctypes.c_size_t


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run python -m paper_2605_06675_gb300.build")
        L = ctypes.CDLL(LIB_PATH)
        sig = {
            "rq_status_string": ([_I], ctypes.c_char_p),
            "rq_abi_version": ([], _I),
            "rq_lloydmax_levels": ([_I, _P], _I),
            "rq_fit_distortion": ([_I, _P, _I, _I, _D, _P, _P, _P, _P], _I),
            "rq_alloc": ([_I, _P, _P, _P, _D, _U, _U, _P, _P], _I),
            "rq_alloc_continuous": ([_I, _P, _P, _P, _D, _D, _D, _P], _I),
            "rq_packed_layout": ([_P, _P, _P, _P], _I),
            "rq_calibrate_workspace_bytes": ([_I, _I], _SZ),
            "rq_calibrate_distortion": ([_P, _I, _I, _I, _I, _I, _I, _I, _I, _P, _P, _P, _SZ, _P,
                                         _P], _I),
            "rq_quantize_pack": ([_P, _I, _P, _P, _P, _P, _P, _P, _P, _P], _I),
            "rq_decode_workspace_bytes": ([_P, _P], _I),
            "rq_decode_attention": ([_P, _I, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P], _I),
            "rq_decode_attention_static": ([_P, _I, _P, _P, _P, _P, _P, _P, _P, _P], _I),
            "rq_residual_bytes": ([_P], _SZ),
            "rq_append": ([_P, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P], _I),
            "rq_decode_attention_len": ([_P, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P],
                                        _I),
            "rq_append_rows": ([_P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P], _I),
            "rq_decode_attention_rows": ([_P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P],
                                         _I),
            "rq_decode_set_pattern": ([_I], _I),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _check(fn: str, status: int) -> None:
    if status != RQ_OK:
        raise RQError(fn, status)


def _host(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


def _hp(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dp(t):
    """Device pointer of a CUDA tensor (or None)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return ctypes.c_void_p(t.data_ptr())


def _dp_readable(t):
    """Pointer the device can read: a CUDA tensor, or a pinned (page-locked)
    host tensor, whose address the device uses directly under unified
    addressing (the kernel then reads it over the host link)."""
    if t is not None and not t.is_cuda:
        if not t.is_pinned():
            raise ValueError("expected a CUDA tensor or a pinned host tensor")
        if not t.is_contiguous():
            raise ValueError("expected a contiguous tensor")
        return ctypes.c_void_p(t.data_ptr())
    return _dp(t)


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def torch_dtype_code(dtype) -> int:
    import torch
    if dtype == torch.float16:
        return RQ_F16
    if dtype == torch.bfloat16:
        return RQ_BF16
    raise ValueError(f"unsupported dtype {dtype}")


def make_desc(L, B, H_kv, H_q, S, dtype, k_grouping, v_grouping, hadamard=False,
              k_quantizer=RQ_MINMAX, v_quantizer=RQ_MINMAX) -> rq_cache_desc:
    code = dtype if isinstance(dtype, int) else torch_dtype_code(dtype)
    return rq_cache_desc(L, B, H_kv, H_q, S, HEAD_DIM, GROUP, code, k_grouping, v_grouping,
                         1 if hadamard else 0, k_quantizer, v_quantizer)


# ------------------------------------------------------------------ host ----

def rq_status_string(status: int) -> str:
    return lib().rq_status_string(status).decode()


def rq_abi_version() -> int:
    return lib().rq_abi_version()


def rq_lloydmax_levels(b: int) -> np.ndarray:
    """The library's fp16 Lloyd-Max codebook at b bits (2^b levels, ascending)."""
    out = np.zeros(2 ** b, dtype=np.uint16)
    _check("rq_lloydmax_levels", lib().rq_lloydmax_levels(b, _hp(out)))
    return out.view(np.float16)


def rq_fit_distortion(mse, b_lo=2, b_hi=6, r2_min=0.96, classes=None):
    mse = _host(mse, np.float64)
    n = mse.shape[0]
    assert mse.shape == (n, 8)
    alpha = np.zeros(n)
    beta = np.zeros(n)
    r2 = np.zeros(n)
    cls = None if classes is None else _host(classes, np.int32)
    _check("rq_fit_distortion", lib().rq_fit_distortion(
        n, _hp(mse), b_lo, b_hi, r2_min, None if cls is None else _hp(cls),
        _hp(alpha), _hp(beta), _hp(r2)))
    return alpha, beta, r2


def rq_alloc(w, alpha, beta, avg_bits, allowed_mask, flags=0):
    w = _host(w, np.float64)
    alpha = _host(alpha, np.float64)
    beta = _host(beta, np.float64)
    n = w.shape[0]
    bits = np.zeros(n, dtype=np.uint8)
    obj = ctypes.c_double(0.0)
    _check("rq_alloc", lib().rq_alloc(n, _hp(w), _hp(alpha), _hp(beta), float(avg_bits),
                                      int(allowed_mask), int(flags), _hp(bits),
                                      ctypes.byref(obj)))
    return bits, obj.value


def rq_alloc_continuous(w, alpha, beta, avg_bits, b_min, b_max):
    w = _host(w, np.float64)
    alpha = _host(alpha, np.float64)
    beta = _host(beta, np.float64)
    n = w.shape[0]
    out = np.zeros(n)
    _check("rq_alloc_continuous", lib().rq_alloc_continuous(
        n, _hp(w), _hp(alpha), _hp(beta), float(avg_bits), float(b_min), float(b_max), _hp(out)))
    return out


def rq_packed_layout(desc: rq_cache_desc, bits):
    bits = _host(bits, np.uint8).reshape(desc.L, desc.H_kv, 2)
    offsets = np.zeros((desc.L, desc.B, desc.H_kv, 2), dtype=np.uint64)
    total = ctypes.c_uint64(0)
    _check("rq_packed_layout", lib().rq_packed_layout(ctypes.byref(desc), _hp(bits), _hp(offsets),
                                                      ctypes.byref(total)))
    return offsets, total.value


# ---------------------------------------------------------------- device ----

def rq_calibrate_workspace_bytes(n: int, T: int) -> int:
    return lib().rq_calibrate_workspace_bytes(n, T)


def rq_calibrate_distortion(x, k_grouping, v_grouping, hadamard, signs, mse, ws, status=None,
                            stream=None, k_quantizer=RQ_MINMAX, v_quantizer=RQ_MINMAX):
    """x: CUDA [n][T][128] fp16/bf16; mse: CUDA float64 [n][8]; ws: CUDA byte buffer."""
    n, T, d = x.shape
    _check("rq_calibrate_distortion", lib().rq_calibrate_distortion(
        _dp(x), torch_dtype_code(x.dtype), n, T, k_grouping, v_grouping, 1 if hadamard else 0,
        k_quantizer, v_quantizer, _dp(signs), _dp(mse), _dp(ws), ws.numel() * ws.element_size(), _dp(status),
        _stream(stream)))


def rq_quantize_pack(desc, layer, k, v, signs, bits_dev, offsets_dev, packed, status=None,
                     stream=None):
    """k, v: CUDA tensors, or pinned host tensors read by the kernel in place."""
    _check("rq_quantize_pack", lib().rq_quantize_pack(
        ctypes.byref(desc), layer, _dp_readable(k), _dp_readable(v), _dp(signs), _dp(bits_dev),
        _dp(offsets_dev), _dp(packed), _dp(status), _stream(stream)))


def rq_decode_workspace_bytes(desc) -> int:
    out = ctypes.c_size_t(0)
    _check("rq_decode_workspace_bytes", lib().rq_decode_workspace_bytes(ctypes.byref(desc),
                                                                        ctypes.byref(out)))
    return out.value


def rq_decode_attention(desc, layer, q, packed, bits_dev, offsets_dev, signs, out, ws,
                        status=None, stream=None):
    _check("rq_decode_attention", lib().rq_decode_attention(
        ctypes.byref(desc), layer, _dp(q), _dp(packed), _dp(bits_dev), _dp(offsets_dev),
        _dp(signs), _dp(out), _dp(ws), ws.numel() * ws.element_size(), _dp(status),
        _stream(stream)))


def rq_decode_set_pattern(pattern: int) -> None:
    """How this process issues decode calls: RQ_DECODE_BACK_TO_BACK (the
    default; calls follow one another on the stream) or RQ_DECODE_INTERLEAVED
    (other kernels run between them). Sets how the split kernel deals splits
    to its CTAs and where the merge CTAs start; results are bit-identical
    either way."""
    _check("rq_decode_set_pattern", lib().rq_decode_set_pattern(pattern))


def rq_decode_attention_static(desc, layer, q, packed, bits_dev, offsets_dev, signs, out,
                               status=None, stream=None):
    """rq_decode_attention without a workspace argument: for callers that
    cannot allocate device memory where they decode (runtimes whose allocator
    belongs to someone else, plugins handed only their inputs and outputs).
    Uses librq's fixed RQ_STATIC_SCRATCH_BYTES device array, shared by every
    call on the device, so concurrent calls on unordered streams race."""
    _check("rq_decode_attention_static", lib().rq_decode_attention_static(
        ctypes.byref(desc), layer, _dp(q), _dp(packed), _dp(bits_dev), _dp(offsets_dev),
        _dp(signs), _dp(out), _dp(status), _stream(stream)))


def rq_residual_bytes(desc) -> int:
    return int(lib().rq_residual_bytes(ctypes.byref(desc)))


def rq_append(desc, layer, pos, k_new, v_new, residual, signs, bits_dev, offsets_dev, packed,
              status=None, stream=None):
    """Append token ``pos`` (k_new, v_new: CUDA [B][H_kv][128]) of one layer to
    the residual windows; a full window is quantized into block pos // 32."""
    _check("rq_append", lib().rq_append(
        ctypes.byref(desc), layer, pos, _dp(k_new), _dp(v_new), _dp(residual), _dp(signs),
        _dp(bits_dev), _dp(offsets_dev), _dp(packed), _dp(status), _stream(stream)))


def rq_decode_attention_len(desc, layer, n_tokens, q, packed, bits_dev, offsets_dev, signs,
                            residual, out, ws, status=None, stream=None):
    """Decode attention over the first ``n_tokens`` tokens: packed blocks plus
    the residual window's last n_tokens % 32 tokens."""
    _check("rq_decode_attention_len", lib().rq_decode_attention_len(
        ctypes.byref(desc), layer, n_tokens, _dp(q), _dp(packed), _dp(bits_dev),
        _dp(offsets_dev), _dp(signs), _dp(residual), _dp(out), _dp(ws),
        ws.numel() * ws.element_size(), _dp(status), _stream(stream)))


def rq_append_rows(desc, layer, pos, k_new, v_new, residual, signs, bits_dev, offsets_dev, packed,
                   status=None, stream=None):
    """Append one token per batch row at the rows' own positions (``pos``:
    CUDA int32 [B]; a negative entry appends nothing for that row)."""
    _check("rq_append_rows", lib().rq_append_rows(
        ctypes.byref(desc), layer, _dp(pos), _dp(k_new), _dp(v_new), _dp(residual), _dp(signs),
        _dp(bits_dev), _dp(offsets_dev), _dp(packed), _dp(status), _stream(stream)))


def rq_decode_attention_rows(desc, layer, n_tokens, q, packed, bits_dev, offsets_dev, signs,
                             residual, out, ws, status=None, stream=None):
    """Decode attention with a token count per batch row (``n_tokens``: CUDA
    int32 [B])."""
    _check("rq_decode_attention_rows", lib().rq_decode_attention_rows(
        ctypes.byref(desc), layer, _dp(n_tokens), _dp(q), _dp(packed), _dp(bits_dev),
        _dp(offsets_dev), _dp(signs), _dp(residual), _dp(out), _dp(ws),
        ws.numel() * ws.element_size(), _dp(status), _stream(stream)))
