"""rq_quantize_pack reading K and V from pinned host memory.

The quantize kernel accepts any K/V pointer the device can address; given
page-locked host tensors it reads them over the host link with no staging
copy. The packed cache must equal, byte for byte, the one packed from the same
values in device memory, and the decode over it must match the oracle. A host
tensor that is not pinned is refused by the binding."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle, ensure_built
from .test_gpu_parity import check_layer

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


@pytest.mark.parametrize("kg,hadamard,dtype", [(PER_CHANNEL, False, "bfloat16"),
                                               (PER_TOKEN, True, "float16")])
def test_pinned_host_kv_packs_identically(kg, hadamard, dtype):
    ensure_built()
    wl = Workload("hostkv", L=2, B=2, H_kv=4, H_q=16, S=32 * 37, dtype=dtype, k_grouping=kg,
                  v_grouping=PER_TOKEN, hadamard=hadamard, allowed=(2, 3, 4, 5, 8), avg_bits=3.5,
                  sigma_lnw=0.5, value_dist="gaussian", seed=83)
    signs = synth.hadamard_signs(wl.seed) if hadamard else None
    bits = bits_cycle(wl.L, wl.H_kv, wl.allowed)
    dev_path = PackedKVPath(wl, DEV, signs)
    dev_path.set_bits(bits)
    host_path = PackedKVPath(wl, DEV, signs)
    host_path.set_bits(bits)
    dev_path.packed.zero_()                 # layers not yet packed compare as zeros
    host_path.packed.zero_()
    for l in range(wl.L):
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, device=DEV)
        hk, hv = k.cpu().pin_memory(), v.cpu().pin_memory()
        dev_path.quantize(l, k, v)
        host_path.quantize(l, hk, hv)
        torch.cuda.synchronize()
        assert torch.equal(host_path.packed[:host_path.total_bytes],
                           dev_path.packed[:dev_path.total_bytes]), l
    assert int(host_path.status.item()) == 0
    # the decode over the host-packed cache against the oracle (layer 1)
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, 1, device=DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, 1, DEV)
    out = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    host_path.decode(1, q, out)
    torch.cuda.synchronize()
    check_layer(host_path, wl, 1, k, v, q, out, signs)


def test_unpinned_host_kv_is_refused():
    rq = ensure_built()
    wl = Workload("hostkv2", L=1, B=1, H_kv=2, H_q=8, S=64, dtype="bfloat16",
                  k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                  allowed=(2, 3, 4), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian", seed=84)
    path = PackedKVPath(wl, DEV)
    path.set_bits(np.full((1, 2, 2), 3, dtype=np.uint8))
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, 0)
    with pytest.raises(ValueError):          # the binding
        path.quantize(0, k, v)
    # the C ABI itself: pageable host memory is refused before any launch
    st = rq.lib().rq_quantize_pack(ctypes.byref(path.desc), 0, ctypes.c_void_p(k.data_ptr()),
                                   ctypes.c_void_p(v.data_ptr()), None,
                                   ctypes.c_void_p(path.bits.data_ptr()),
                                   ctypes.c_void_p(path.offsets.data_ptr()),
                                   ctypes.c_void_p(path.packed.data_ptr()),
                                   ctypes.c_void_p(path.status.data_ptr()), None)
    assert rq.STATUS_NAMES[st] == "RQ_ERR_INVALID_ARG"
    torch.cuda.synchronize()
    assert int(path.status.item()) == 0
