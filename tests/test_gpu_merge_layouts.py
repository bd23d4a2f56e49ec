"""The two launch layouts of the decode merge.

When a call's merge grid has at most one CTA per SM and its shared memory
fits beside the split CTAs, the split kernel runs at 120 registers a thread
and the merge CTAs start beside the split CTAs, waiting there for the split
grid to end; otherwise the split kernel runs at 128 registers and the merge
CTAs start where split CTAs have left. These tests put shapes on both sides
of that line (KIVI and rotated caches, GQA 4 and 8, residual tokens, ragged
rows) and check them against the oracle, and check that calls of either
layout issued back to back equal the same calls made alone."""
import pytest
import torch

from oracle import pipeline as opipe
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300.path import PackedKVPath
from paper_2605_06675_gb300.workloads import PER_CHANNEL, PER_TOKEN, Workload

from .gpu_helpers import TOL, attn_err, bits_cycle, ensure_built, oracle_layer, to_np
from .test_gpu_parity import check_layer

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
GROUP_BYTES = 52480        # shared memory of one split group
RESERVED = 1024            # shared memory the device reserves per CTA
MERGE_STATIC = {1: 8320, 2: 4224, 4: 4224, 8: 4224}   # the merge kernel's static shared memory


def _plan_splits(units, nblk):
    """Splits per unit of the library's plan (the larger of its two counts)."""
    slots = torch.cuda.get_device_properties(0).multi_processor_count * 4

    def even(sp):
        sp = max(1, min(sp, nblk))
        bps = max(1, -(-nblk // sp))
        return max(1, -(-nblk // bps))

    sp = slots // units
    s = even(sp)
    if units <= slots and slots % units and sp < nblk:
        s = max(s, even(sp + 1))
    return s


def _co_resident(wl, nblk=None, residual=False):
    """The library's layout choice for one call, restated."""
    props = torch.cuda.get_device_properties(0)
    sms = props.multi_processor_count
    smem_sm = getattr(props, "shared_memory_per_multiprocessor", 233472)
    units, g = wl.B * wl.H_kv, wl.H_q // wl.H_kv
    if units > sms:
        return False
    splits = _plan_splits(units, wl.S // 32 if nblk is None else nblk)
    cq = 1 if wl.hadamard else 8
    while cq > 1 and units * cq > sms:
        cq //= 2
    msm = g * splits * (128 // cq // 4 + 1) * 16
    if residual:
        msm = max(msm, 38016)
    msm = min(msm, 65536)
    G = 4 if g <= 4 else 1
    left = smem_sm - (4 // G) * (G * GROUP_BYTES + RESERVED)
    return MERGE_STATIC[cq] + msm + RESERVED <= left


def _wl(name, B, H, g, S, kg=PER_CHANNEL, hadamard=False, seed=0, L=1):
    return Workload(name, L=L, B=B, H_kv=H, H_q=H * g, S=S, dtype="bfloat16", k_grouping=kg,
                    v_grouping=PER_TOKEN, hadamard=hadamard,
                    allowed=(2, 3, 4, 8) if kg == PER_CHANNEL else (3, 4, 5, 6), avg_bits=3.0,
                    sigma_lnw=0.5, value_dist="gaussian", seed=seed)


# (name, B, H_kv, g, S, key grouping, rotated, co-resident merge)
CASES = [
    ("co_g4", 16, 8, 4, 32 * 24, PER_CHANNEL, False, True),      # 128 units, two parts
    ("co_rot", 16, 8, 4, 32 * 24, PER_TOKEN, True, True),        # whole rows
    ("co_g8", 4, 8, 8, 32 * 20, PER_CHANNEL, False, True),       # one-group CTAs
    ("co_few", 2, 4, 4, 32 * 40, PER_CHANNEL, False, True),      # 8 units, eight parts
    ("late_g4", 1, 4, 4, 32 * 200, PER_CHANNEL, False, False),   # many records per unit
    ("late_g8", 8, 8, 8, 32 * 40, PER_CHANNEL, False, False),    # GQA 8, 64 units
    ("late_rot", 2, 2, 4, 32 * 120, PER_TOKEN, True, False),
    ("late_units", 40, 4, 4, 32 * 8, PER_CHANNEL, False, False),  # more units than SMs
]


def _setup(wl, layer=0):
    signs = synth.hadamard_signs(wl.seed).to(DEV) if wl.hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    path.set_bits(bits_cycle(wl.L, wl.H_kv, wl.allowed, offset=wl.seed))
    k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, layer, device=DEV)
    q = synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, layer, DEV)
    path.quantize(layer, k, v)
    return path, signs, k, v, q


def _sampled_streams(wl):
    rows = sorted({0, wl.B // 2, wl.B - 1})
    return [(b, h) for b in rows for h in range(wl.H_kv)]


@pytest.mark.parametrize("name,B,H,g,S,kg,hadamard,co", CASES)
def test_both_layouts_match_oracle(name, B, H, g, S, kg, hadamard, co):
    ensure_built()
    wl = _wl(name, B, H, g, S, kg, hadamard, seed=len(name) + B)
    assert _co_resident(wl) == co
    path, signs, k, v, q = _setup(wl)
    out = torch.full((wl.B, wl.H_q, 128), float("nan"), dtype=torch.float32, device=DEV)
    path.decode(0, q, out)
    torch.cuda.synchronize()
    assert int(path.status.item()) == 0
    assert torch.isfinite(out).all()
    check_layer(path, wl, 0, k, v, q, out, signs, streams=_sampled_streams(wl))


@pytest.mark.parametrize("name,B,H,g,S,kg,hadamard,co", [c for c in CASES if c[0] != "late_units"])
def test_both_layouts_back_to_back(name, B, H, g, S, kg, hadamard, co):
    """Four layers decoded three times over with no host sync in between
    equal each layer decoded alone."""
    ensure_built()
    wl = _wl(name, B, H, g, S, kg, hadamard, seed=11, L=4)
    assert _co_resident(wl) == co
    signs = synth.hadamard_signs(wl.seed).to(DEV) if hadamard else None
    path = PackedKVPath(wl, DEV, signs)
    path.set_bits(bits_cycle(wl.L, wl.H_kv, wl.allowed))
    Q = []
    for l in range(wl.L):
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, device=DEV)
        path.quantize(l, k, v)
        Q.append(synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, l, DEV))
    path.decode_workspace()
    torch.cuda.synchronize()
    outs = [torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=DEV) for _ in range(wl.L)]
    for _ in range(3):
        for l in range(wl.L):
            path.decode(l, Q[l], outs[l])
    torch.cuda.synchronize()
    for l in range(wl.L):
        alone = torch.empty_like(outs[l])
        path.decode(l, Q[l], alone)
        torch.cuda.synchronize()
        assert torch.equal(outs[l], alone), l
    assert int(path.status.item()) == 0


@pytest.mark.parametrize("name,B,H,g,S", [
    ("pat_g4", 16, 4, 4, 32 * 38),     # 64 units: splits of two sizes, four-group CTAs
    ("pat_g8", 4, 8, 8, 32 * 40),      # one-group CTAs
    ("pat_late", 1, 4, 4, 32 * 200),   # the late merge layout
])
def test_call_patterns_are_bit_identical(name, B, H, g, S):
    """RQ_DECODE_INTERLEAVED deals every CTA one split from each quarter of
    the plan and starts the merge CTAs where split CTAs have left (128
    registers), RQ_DECODE_BACK_TO_BACK deals consecutive splits and, where it
    fits, starts them beside the split CTAs: the same splits and the same
    arithmetic either way, so the same output, bit for bit."""
    rq = ensure_built()
    wl = _wl(name, B, H, g, S, seed=13)
    path, signs, k, v, q = _setup(wl)
    outs = []
    try:
        for pattern in (rq.RQ_DECODE_BACK_TO_BACK, rq.RQ_DECODE_INTERLEAVED):
            rq.rq_decode_set_pattern(pattern)
            out = torch.full((wl.B, wl.H_q, 128), float("nan"), dtype=torch.float32, device=DEV)
            path.decode(0, q, out)
            torch.cuda.synchronize()
            outs.append(out)
    finally:
        rq.rq_decode_set_pattern(rq.RQ_DECODE_BACK_TO_BACK)
    assert int(path.status.item()) == 0
    assert torch.isfinite(outs[0]).all()
    assert torch.equal(outs[0], outs[1])
    check_layer(path, wl, 0, k, v, q, outs[1], signs, streams=_sampled_streams(wl))


@pytest.mark.parametrize("late", [False, True])
def test_residual_tokens_both_layouts(late):
    """decode_len over a packed prefix plus raw tokens in the residual
    windows. The residual record needs 38 KB of merge shared memory, so these
    calls merge late whatever the shape; a shape that is co-resident without
    residual tokens is checked too."""
    ensure_built()
    if late:
        wl, n = _wl("res_late", 1, 2, 4, 32 * 100, seed=6), 32 * 90 + 21
    else:
        wl, n = _wl("res_co", 16, 4, 4, 32 * 20, seed=5), 32 * 18 + 13
    s_pk = 32 * (n // 32)
    assert _co_resident(wl, n // 32) == (not late)
    assert not _co_resident(wl, n // 32, residual=True)
    path, signs, k, v, q = _setup(wl)
    for pos in range(s_pk, n):        # the open window's tokens
        path.append(0, pos, k[:, :, pos].contiguous(), v[:, :, pos].contiguous())
    out = torch.full((wl.B, wl.H_q, 128), float("nan"), dtype=torch.float32, device=DEV)
    path.decode_len(0, n, q, out)
    torch.cuda.synchronize()
    assert int(path.status.item()) == 0
    ol = oracle_layer(k[:, :, :s_pk], v[:, :, :s_pk], path.bits_host[0], wl.k_grouping,
                      wl.v_grouping, wl.hadamard, signs)
    ref = opipe.attend_with_residual(to_np(q), ol, to_np(k[:, :, s_pk:n]), to_np(v[:, :, s_pk:n]))
    err = attn_err(to_np(out), ref)
    assert err <= TOL, err
    # the same cache over whole blocks only (no residual tokens)
    path.decode_len(0, s_pk, q, out)
    torch.cuda.synchronize()
    ref = opipe.attend_with_residual(to_np(q), ol, to_np(k[:, :, s_pk:s_pk]),
                                     to_np(v[:, :, s_pk:s_pk]))
    assert attn_err(to_np(out), ref) <= TOL
    assert int(path.status.item()) == 0
