"""rq_decode_attention_static: decode attention for callers that cannot
allocate device memory where they decode (runtimes whose device allocator
belongs to someone else, plugins handed only their inputs and outputs). Its
split-K partial records live in librq's fixed device array instead of a
caller workspace. Checked through the C ABI against
rq_decode_attention: the same kernel on the same inputs, so the outputs must
be bit-identical. The calls come in a row on the shared array: first a
larger shape (more records per (batch, kv head), more of the array written),
then smaller ones that find its leftovers. This file is collected last on
purpose."""
import pytest
import torch

from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import bits_cycle, ensure_built

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _workload(B, S, seed):
    return Workload(f"noalloc{seed}", L=2, B=B, H_kv=4, H_q=16, S=S, dtype="bfloat16",
                    k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                    allowed=(2, 3, 4, 8), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian",
                    seed=seed)


def _both(rq, wl, layer, q_seed):
    """(static output, workspace output) of one layer."""
    path = PackedKVPath(wl, DEV)
    path.set_bits(bits_cycle(wl.L, wl.H_kv, wl.allowed))
    ws = path.decode_workspace()
    assert ws.numel() <= rq.RQ_STATIC_SCRATCH_BYTES
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, layer, device=DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed + q_seed, layer, DEV)
    path.quantize(layer, k, v)
    ref = torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV)
    out = torch.full((wl.B, wl.H_q, 128), float("nan"), dtype=torch.float32, device=DEV)
    rq.rq_decode_attention(path.desc, layer, q, path.packed, path.bits, path.offsets, None,
                           ref, ws, path.status)
    rq.rq_decode_attention_static(path.desc, layer, q, path.packed, path.bits, path.offsets,
                                  None, out, path.status)
    torch.cuda.synchronize()
    assert int(path.status.item()) == 0
    return out, ref


def test_static_scratch_matches_workspace_version():
    rq = ensure_built()
    # a large call first: 4 x 4 (batch, kv head) units over 8192 tokens take
    # several records each; then two smaller calls (fewer units and records)
    # run on what it left in the shared array
    calls = [(_workload(4, 8192, 41), 1, 0), (_workload(3, 2048, 42), 0, 0),
             (_workload(3, 2048, 42), 1, 1)]
    for wl, layer, q_seed in calls:
        out, ref = _both(rq, wl, layer, q_seed)
        assert torch.isfinite(out).all()
        assert torch.equal(out, ref), wl.name


def test_static_scratch_rejects_oversized_shapes():
    rq = ensure_built()
    # counters and records beyond the fixed array: refused on the host before
    # any launch
    big = rq.make_desc(1, 256, 8, 64, 32 * 4096, torch.bfloat16, PER_CHANNEL, PER_TOKEN)
    need = rq.rq_decode_workspace_bytes(big)
    assert need > rq.RQ_STATIC_SCRATCH_BYTES
    dummy = torch.zeros(16, dtype=torch.uint8, device=DEV)
    q = torch.zeros((256, 64, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.zeros((256, 64, 128), dtype=torch.float32, device=DEV)
    bits = torch.full((1, 8, 2), 2, dtype=torch.uint8, device=DEV)
    offs = torch.zeros((1, 256, 8, 2), dtype=torch.int64, device=DEV)
    with pytest.raises(rq.RQError) as e:
        rq.rq_decode_attention_static(big, 0, q, dummy, bits, offs, None, out)
    assert e.value.status == 5
