"""Decode split plans at the edges of one wave.

The plan fills one wave of resident splits (SMs x 4): every (batch, kv head)
unit takes slots / units splits, some one more when the units do not divide
the slots, and a CTA holds four split groups when g <= 4 (one otherwise). These
cases put the unit count below, at and above the wave: more units than slots
(one split per unit, a grid of several waves whose last CTA is part-filled),
a few units short of the slots (almost every unit at one split, the rest at
two), and tiny units (one or two blocks). Every case is checked against the
oracle on a sample of streams, plus bit-identity with the allocation-free
entry point where the workspace fits its array."""
import pytest
import torch

from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle, ensure_built
from .test_gpu_parity import check_layer

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


def _slots():
    props = torch.cuda.get_device_properties(0)
    return props.multi_processor_count * 4


@pytest.mark.parametrize("g", [4, 8])
@pytest.mark.parametrize("units_vs_slots,S", [(+8, 64), (-8, 96), (0, 32 * 5), (+3, 32)])
def test_plan_edges_match_oracle(g, units_vs_slots, S):
    rq = ensure_built()
    H = 8
    B = max(1, (_slots() + units_vs_slots) // H)
    wl = Workload(f"plan{g}{units_vs_slots}", L=1, B=B, H_kv=H, H_q=H * g, S=S, dtype="bfloat16",
                  k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                  allowed=(2, 3, 4, 8), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian",
                  seed=91 + g)
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits_cycle(1, H, wl.allowed, offset=g))
    k, v = synth.kv_layer(B, H, S, wl.dtype, wl.seed, 0, device=DEV)
    q = synth.queries(B, wl.H_q, wl.dtype, wl.seed, 0, DEV)
    out = torch.empty((B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    path.quantize(0, k, v)
    path.decode(0, q, out)
    torch.cuda.synchronize()
    assert int(path.status.item()) == 0
    # the first, a middle and the last batch rows, every head
    rows = sorted({0, B // 2, B - 1})
    check_layer(path, wl, 0, k, v, q, out, None, streams=[(b, h) for b in rows for h in range(H)])
    if rq.rq_decode_workspace_bytes(path.desc) <= rq.RQ_STATIC_SCRATCH_BYTES:
        st = torch.full_like(out, float("nan"))
        rq.rq_decode_attention_static(path.desc, 0, q, path.packed, path.bits, path.offsets, None,
                                      st, path.status)
        torch.cuda.synchronize()
        assert torch.equal(st, out)
