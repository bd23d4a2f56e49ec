"""The C-ABI calls inside a captured CUDA graph.

Quantize + pack of every layer and decode attention of every layer are
captured once on a side stream and replayed; the packed cache and the outputs
must equal those of the same calls launched one by one, bit for bit. A new
allocation written by set_bits (in place, same table shapes) must be picked
up by the next replay without capturing again."""
import numpy as np
import pytest
import torch

from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle, ensure_built

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


def _eager(path, wl, K, V, Q):
    out = [torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV) for _ in range(wl.L)]
    path.packed.zero_()
    for l in range(wl.L):
        path.quantize(l, K[l], V[l])
    for l in range(wl.L):
        path.decode(l, Q[l], out[l])
    torch.cuda.synchronize()
    return path.packed.clone(), [o.clone() for o in out]


@pytest.mark.gpu
@pytest.mark.parametrize("kg,vg,hadamard,allowed", [
    (PER_CHANNEL, PER_TOKEN, False, (2, 3, 4, 8)),      # KIVI layout (compile-time loops)
    (PER_TOKEN, PER_TOKEN, True, (3, 4, 5, 6)),         # rotated per-token (both decode paths)
])
def test_graph_replay_equals_launches(kg, vg, hadamard, allowed):
    ensure_built()
    wl = Workload("graphs", L=3, B=2, H_kv=4, H_q=16, S=256, dtype="bfloat16", k_grouping=kg,
                  v_grouping=vg, hadamard=hadamard, allowed=allowed, avg_bits=4.0,
                  sigma_lnw=0.5, value_dist="gaussian", seed=61)
    signs = synth.hadamard_signs(wl.seed).to(DEV) if hadamard else None
    K, V, Q = [], [], []
    for l in range(wl.L):
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, device=DEV)
        K.append(k)
        V.append(v)
        Q.append(synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, l, DEV))
    cap = wl.L * wl.B * wl.H_kv * 2 * (wl.S // 32) * 512 * (max(allowed) + 1)
    tables = [bits_cycle(wl.L, wl.H_kv, allowed, offset=o) for o in (0, 1)]

    path = PackedKVPath(wl, DEV, signs)
    path.set_bits(tables[0], capacity=cap)
    path.decode_workspace()
    bits_ptr = path.bits.data_ptr()
    want = []
    for t in tables:
        path.set_bits(t, capacity=cap)
        want.append(_eager(path, wl, K, V, Q))
    assert path.bits.data_ptr() == bits_ptr          # tables updated in place

    out = [torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV) for _ in range(wl.L)]
    stream = torch.cuda.Stream(DEV)
    path.set_bits(tables[0], capacity=cap)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for l in range(wl.L):
            path.quantize(l, K[l], V[l])
        for l in range(wl.L):
            path.decode(l, Q[l], out[l])
    for t, (packed, outs) in zip(tables, want):
        path.set_bits(t, capacity=cap)
        path.packed.zero_()
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(path.packed, packed)
        for l in range(wl.L):
            assert torch.equal(out[l], outs[l]), l
    assert int(path.status.item()) == 0
    assert np.array_equal(path.bits.cpu().numpy(), tables[1])
