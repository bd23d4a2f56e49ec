"""Decode calls issued back to back on one workspace.

A decode call's split grid may start while the previous call's merge grid is
still reading the split records from the shared workspace; it must not write
its own records until that merge has finished. The shapes here make the race
window wide: two (batch, kv head) units share the wave, so every unit has
hundreds of splits of one or two blocks each (the split grid reaches its
record writes within a few microseconds) while the merge pulls hundreds of
records per query row in several round trips. Each back-to-back output must
equal, bit for bit, the same call made alone, and one layer is checked against
the oracle."""
import pytest
import torch

from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle, ensure_built
from .test_gpu_parity import check_layer

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


@pytest.mark.parametrize("g,kg,hadamard", [
    (4, PER_CHANNEL, False),      # four split groups per CTA, KIVI layout
    (8, PER_CHANNEL, False),      # one split group per CTA (g = 8)
    (4, PER_TOKEN, True),         # rotated per-token cache (whole-row merge)
])
def test_back_to_back_equals_alone(g, kg, hadamard):
    ensure_built()
    wl = Workload(f"b2b{g}{kg}", L=6, B=1, H_kv=2, H_q=2 * g, S=32 * 640, dtype="bfloat16",
                  k_grouping=kg, v_grouping=PER_TOKEN, hadamard=hadamard,
                  allowed=(2, 3, 4, 8) if kg == PER_CHANNEL else (3, 4, 5, 6), avg_bits=3.5,
                  sigma_lnw=0.5, value_dist="gaussian", seed=71 + g)
    signs = synth.hadamard_signs(wl.seed).to(DEV) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    path.set_bits(bits_cycle(wl.L, wl.H_kv, wl.allowed))
    K, V, Q = [], [], []
    for l in range(wl.L):
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, device=DEV)
        K.append(k)
        V.append(v)
        Q.append(synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, l, DEV))
        path.quantize(l, k, v)
    path.decode_workspace()
    torch.cuda.synchronize()

    outs = [torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV) for _ in range(wl.L)]
    for rep in range(3):                         # back to back, no host sync in between
        for l in range(wl.L):
            path.decode(l, Q[l], outs[l])
    torch.cuda.synchronize()
    for l in range(wl.L):
        alone = torch.empty_like(outs[l])
        path.decode(l, Q[l], alone)
        torch.cuda.synchronize()
        assert torch.equal(outs[l], alone), f"layer {l}"
    assert int(path.status.item()) == 0
    check_layer(path, wl, 0, K[0], V[0], Q[0], outs[0], signs)
