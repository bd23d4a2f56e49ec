"""Host-side behaviour of PackedKVPath that needs no GPU: set_bits lays out
the packed cache with the library's host call and rewrites the width and
offset tables in place (so work captured in a CUDA graph sees the new
allocation)."""
import numpy as np
import torch

from paper_2605_06675_gb300 import rq
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle


def _wl():
    return Workload("path_host", L=2, B=3, H_kv=4, H_q=8, S=96, dtype="bfloat16",
                    k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                    allowed=(2, 3, 4, 8), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian",
                    seed=71)


def test_set_bits_rewrites_tables_in_place():
    wl = _wl()
    path = PackedKVPath(wl, "cpu")
    a = bits_cycle(wl.L, wl.H_kv, wl.allowed, offset=0)
    b = bits_cycle(wl.L, wl.H_kv, wl.allowed, offset=1)
    path.set_bits(a, capacity=1 << 20)
    bits_ptr, offs_ptr, packed_ptr = path.bits.data_ptr(), path.offsets.data_ptr(), path.packed.data_ptr()
    offsets_b, total_b = path.set_bits(b, capacity=1 << 20)
    assert path.bits.data_ptr() == bits_ptr
    assert path.offsets.data_ptr() == offs_ptr
    assert path.packed.data_ptr() == packed_ptr          # capacity unchanged: no new buffer
    assert np.array_equal(path.bits.numpy(), b)
    assert np.array_equal(path.offsets.numpy(), offsets_b.view(np.int64))
    ref_offsets, ref_total = rq.rq_packed_layout(path.desc, b)
    assert np.array_equal(offsets_b, ref_offsets) and total_b == ref_total


def test_set_bits_layout_is_prefix_sum_of_stream_bytes():
    # stream (l, batch, h, kind) holds S/32 blocks of 512 (b + 1) bytes, streams
    # laid out in [layer][batch][head][kind] order
    wl = _wl()
    path = PackedKVPath(wl, "cpu")
    bits = bits_cycle(wl.L, wl.H_kv, wl.allowed, offset=3)
    offsets, total = path.set_bits(bits)
    sizes = np.zeros((wl.L, wl.B, wl.H_kv, 2), dtype=np.int64)
    for l in range(wl.L):
        for bb in range(wl.B):
            for h in range(wl.H_kv):
                for kind in range(2):
                    sizes[l, bb, h, kind] = (wl.S // 32) * 512 * (int(bits[l, h, kind]) + 1)
    flat = sizes.reshape(-1)
    starts = np.concatenate([[0], np.cumsum(flat)[:-1]])
    assert np.array_equal(offsets.reshape(-1).astype(np.int64), starts)
    assert total == int(flat.sum())
    assert path.packed.numel() >= total
    assert path.packed.dtype == torch.uint8
