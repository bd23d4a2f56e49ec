#!/usr/bin/env python
"""Benchmark of the RateQuant packed mixed-bit KV path on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
  a1  distortion sweep b = 1..8 on the calibration sample (GPU)
  a2  fit D(b) = alpha beta^-b (host), a3 integer allocation (host) + layout
  a4/a5  quantize + bit-pack every layer of the cache (GPU, one launch/layer)
  a6/a7  split-K decode attention on the packed cache for every layer (GPU)

Prints ONE JSON line (rank 0). ``value`` is the step's algorithmic bytes /
step time (GB/s); the decode-attention and quantize-pack numbers of the
metric are under ``components``. ``--impl reference`` times the CPU oracle
(the only reference that exists: the paper ships no code) on bounded samples.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "packed mixed-bit decode-attention GB/s (% HBM peak), tokens/s; quantize GB/s"
FALLBACK_HBM_GBS = 6800.0


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


QUANTIZERS = ["minmax", "absmax", "lloydmax"]       # rq_quantizer values 0, 1, 2


def _workloads():
    from paper_2605_06675_gb300 import workloads as W
    return {w.name: w for w in W.ALL}, W.LLAMA3_8B_32K


def _parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=None)
    ap.add_argument("--layers", type=int, default=None,
                    help="run only the first N layers (small cases for profiling)")
    ap.add_argument("--k-quantizer", choices=["minmax", "absmax", "lloydmax"], default=None,
                    help="override the workload's key quantizer (absmax = symmetric)")
    ap.add_argument("--v-quantizer", choices=["minmax", "absmax", "lloydmax"], default=None)
    ap.add_argument("--no-graphs", action="store_true",
                    help="launch the per-layer quantize and decode loops one call at a time "
                         "instead of replaying them as CUDA graphs")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-leg", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--cpu-tokens", type=int, default=None, help=argparse.SUPPRESS)
    return ap.parse_args()


# --------------------------------------------------------------------------
# replica timing across ranks (every rank runs the whole path on its own GPU;
# the job's time is the slowest rank's and its value counts every rank's work)
# --------------------------------------------------------------------------

def max_over_ranks(x: float, world: int, device) -> float:
    """Maximum of ``x`` over all ranks of the default process group."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_gbs(world: int, bytes_per_rank_step: float, ms_per_step: float) -> float:
    """Whole-job throughput: every rank's bytes over the slowest rank's time."""
    return world * bytes_per_rank_step / (ms_per_step * 1e-3) / 1e9


# --------------------------------------------------------------------------
# byte accounting (algorithmic bytes; partials and workspaces excluded)
# --------------------------------------------------------------------------

def elem_bytes(wl):
    return 2


def quant_bytes_layer(wl, bits_l):
    """read K and V + write codes and meta of every stream of one layer."""
    nblk = wl.S // 32
    read = 2 * wl.B * wl.H_kv * wl.S * 128 * elem_bytes(wl)
    write = sum(wl.B * nblk * 512 * (int(b) + 1) for b in bits_l.reshape(-1))
    return read + write


def decode_bytes_layer(wl, bits_l):
    """packed codes + meta of every stream + q + fp32 out."""
    nblk = wl.S // 32
    packed = sum(wl.B * nblk * 512 * (int(b) + 1) for b in bits_l.reshape(-1))
    return packed + wl.B * wl.H_q * 128 * elem_bytes(wl) + wl.B * wl.H_q * 128 * 4


def calib_bytes(wl, n, T):
    return n * T * 128 * elem_bytes(wl) + n * 8 * 8


# --------------------------------------------------------------------------
# clocks sampled during the timed region
# --------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.gpu = gpu_index
        self.path = os.path.join("/tmp", f"rq_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.gpu)], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sms, maxs, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sms.append(float(parts[1]))
                maxs.append(float(parts[2]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(nm)
        os.remove(self.path)
        if not sms:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sms), "sm_max_mhz": max(maxs),
                "reasons": sorted(reasons), "samples": len(sms)}


# --------------------------------------------------------------------------
# traffic counters recorded from ncu (valid only for the kernel source they
# were taken on)
# --------------------------------------------------------------------------

def strip_comments(src: str) -> str:
    """C/C++/CUDA source without its comments, whitespace runs collapsed to
    one blank (string and character literals kept as written)."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c == "/" and i + 1 < n and src[i + 1] == "/":
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif c == "/" and i + 1 < n and src[i + 1] == "*":
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        elif c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        else:
            out.append(c)
            i += 1
    return " ".join("".join(out).split())


def kernel_source_hash(name: str) -> str:
    """sha256[:16] of a kernel's translation unit together with the library's
    headers (every .cuh and rq.h), comments stripped: a record goes stale when
    the code of any of them changes, not when a comment does."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_2605_06675_gb300", "csrc")
    h = hashlib.sha256()
    headers = sorted(f for f in os.listdir(csrc) if f.endswith(".cuh"))
    for path in ([os.path.join(csrc, name)] + [os.path.join(csrc, f) for f in headers] +
                 [os.path.join(ROOT, "include", "rq.h")]):
        h.update(strip_comments(open(path, encoding="utf-8").read()).encode())
        h.update(b"\0")
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    for line in open(path):
        if line.startswith("#") or not line.strip():
            continue
        parts = line.split()
        if len(parts) < 4 or parts[0] != kernel or parts[1] != workload:
            continue
        src, want = parts[3].split(":")
        return float(parts[2]) if kernel_source_hash(src) == want else None
    return None


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------

def run_ours(args, wl, rank, world, local_rank):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2605_06675_gb300 import build as _b
    from paper_2605_06675_gb300 import rq, synth
    from paper_2605_06675_gb300.path import PackedKVPath

    if not os.path.exists(_b.LIB):
        if rank == 0:
            _b.build()
        if world > 1:
            dist.barrier()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    # a stream of our own: the per-layer loops are captured as CUDA graphs on it
    stream = torch.cuda.Stream(dev)
    torch.cuda.set_stream(stream)

    # inputs resident in HBM before the timed region
    signs = synth.hadamard_signs(wl.seed) if wl.hadamard else None
    K, V, Q, OUT = [], [], [], []
    for l in range(wl.L):
        k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, wl.value_dist, dev)
        K.append(k)
        V.append(v)
        Q.append(synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, l, dev))
        OUT.append(torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=dev))
    X = synth.calibration_sample(wl, device=dev)
    n, T = X.shape[0], X.shape[1]
    w = synth.importances(n, wl.sigma_lnw, wl.seed)
    path = PackedKVPath(wl, dev, signs)

    # capacity for the packed cache: every stream at the widest allowed width
    cap = wl.L * wl.B * wl.H_kv * 2 * (wl.S // 32) * 512 * (max(wl.allowed) + 1)
    mse0 = path.calibrate(X).cpu().numpy()
    bits0, _ = path.allocate(mse0, w)
    path.set_bits(bits0, capacity=cap)
    path.decode_workspace()
    torch.cuda.synchronize()

    graphs = None

    def step(ev=None, host_ms=None):
        if ev is not None:
            ev[0].record(stream)
        mse = path.calibrate(X)
        if ev is not None:
            ev[1].record(stream)
        mse_h = mse.cpu().numpy()                       # D2H, synchronises
        t0 = time.perf_counter()
        bits, _ = path.allocate(mse_h, w)
        path.set_bits(bits, capacity=cap)
        if host_ms is not None:
            host_ms.append((time.perf_counter() - t0) * 1e3)
        if ev is not None:
            ev[2].record(stream)
        if graphs is not None:
            graphs[0].replay()
        else:
            for l in range(wl.L):
                path.quantize(l, K[l], V[l])
        if ev is not None:
            ev[3].record(stream)
        if graphs is not None:
            graphs[1].replay()
        else:
            for l in range(wl.L):
                path.decode(l, Q[l], OUT[l])
        if ev is not None:
            ev[4].record(stream)
        return bits

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    # The quantize and decode loops of a step as two CUDA graphs (the kernels
    # read the widths and offsets that set_bits writes in place each step).
    launch_mode = "per-layer launches"
    if not args.no_graphs:
        try:
            gq, gd = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
            with torch.cuda.graph(gq, stream=stream):
                for l in range(wl.L):
                    path.quantize(l, K[l], V[l])
            with torch.cuda.graph(gd, stream=stream):
                for l in range(wl.L):
                    path.decode(l, Q[l], OUT[l])
            graphs = (gq, gd)
            launch_mode = "cuda graphs (quantize loop, decode loop)"
            step()
            torch.cuda.synchronize()
        except RuntimeError as e:
            graphs = None
            launch_mode = f"per-layer launches (graph capture failed: {str(e)[:80]})"
            torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]
    host_ms = []
    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.15)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    bits = None
    for i in range(args.steps):
        bits = step(evs[i], host_ms)
    end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    total_ms = max_over_ranks(start.elapsed_time(end), world, dev)
    if world > 1:
        dist.barrier()

    calib_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    quant_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)
    dec_ms = statistics.mean(e[3].elapsed_time(e[4]) for e in evs)
    ms_step = total_ms / args.steps

    qb = sum(quant_bytes_layer(wl, bits[l]) for l in range(wl.L))
    db = sum(decode_bytes_layer(wl, bits[l]) for l in range(wl.L))
    cb = calib_bytes(wl, n, T)
    step_bytes = qb + db + cb
    peak, peak_kind = _peaks()
    value = job_gbs(world, step_bytes, ms_step)
    q_gbs = qb / (quant_ms * 1e-3) / 1e9
    d_gbs = db / (dec_ms * 1e-3) / 1e9
    tok_s = wl.B / (dec_ms * 1e-3)

    # dominant kernel by time share: quantize_pack (per-launch = one layer)
    shares = {"quantize_pack": quant_ms, "decode_attention": dec_ms, "calibrate": calib_ms}
    dom = max(shares, key=shares.get)
    if dom == "quantize_pack":
        per_launch_bytes, per_launch_ms = qb / wl.L, quant_ms / wl.L
        tr = recorded_traffic("quantize_pack", wl.name)
    else:
        per_launch_bytes, per_launch_ms = db / wl.L, dec_ms / wl.L
        tr = recorded_traffic("decode_split", wl.name)
    achieved = per_launch_bytes / (per_launch_ms * 1e-3) / 1e9
    roofline = {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1), "peak": peak,
                "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": tr,
                "algorithmic_bytes_per_launch": int(per_launch_bytes),
                "peak_source": f"{peak_kind} hbm_gbs"}

    result = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16 in; f32 quantizer; f16 x f16 -> f32 mma attention",
        "data": "synthetic (seeded; Llama-3/Qwen3-shaped KV caches, random q)",
        "config": {"workload": wl.name, "L": wl.L, "B": wl.B, "H_kv": wl.H_kv, "H_q": wl.H_q,
                   "S": wl.S, "head_dim": 128, "group": 32, "bits_allowed": list(wl.allowed),
                   "avg_bits": wl.avg_bits, "k_grouping": "per_channel" if wl.k_grouping else "per_token",
                   "v_grouping": "per_channel" if wl.v_grouping else "per_token",
                   "hadamard": wl.hadamard, "k_quantizer": QUANTIZERS[wl.k_quantizer],
                   "v_quantizer": QUANTIZERS[wl.v_quantizer],
                   "calib_tokens": T, "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (no flush)", "launch": launch_mode},
        "components": {
            "decode_attention": {"gbs": round(d_gbs, 1), "frac_of_measured_hbm": round(d_gbs / peak, 4),
                                 "frac_of_8TBs": round(d_gbs / 8000.0, 4),
                                 "tokens_per_s": round(tok_s, 1), "ms_per_step": round(dec_ms, 4),
                                 "bytes_per_step": int(db)},
            "quantize_pack": {"gbs": round(q_gbs, 1), "frac_of_measured_hbm": round(q_gbs / peak, 4),
                              "frac_of_8TBs": round(q_gbs / 8000.0, 4),
                              "ms_per_step": round(quant_ms, 4), "bytes_per_step": int(qb)},
            "calibrate": {"ms_per_step": round(calib_ms, 4), "components": n, "tokens": T},
            "fit_alloc_layout_host": {"ms_per_step": round(statistics.mean(host_ms), 4)},
            "avg_bits_allocated": round(float(bits.mean()), 4),
        },
        "roofline": roofline,
        "clocks": clk,
        "gpu_launches": args.steps * (2 + 3 * wl.L),
    }

    if not args.no_e2e:
        result["e2e"] = run_e2e(args, wl, path, K, V, Q, OUT, X, w, cap, dev, stream,
                                step_bytes, world)
    if rank == 0 and not args.no_cpu_baseline and world == 1:
        result["cpu_baseline"] = run_cpu_leg_subprocess(wl)
    return result


def run_e2e(args, wl, path, K, V, Q, OUT, X, w, cap, dev, stream, step_bytes, world):
    """Same step through the public API with HOST inputs: every step copies
    the calibration sample, each layer's K/V and q from pinned host memory to
    the device and reads every layer's output back."""
    import torch
    import torch.distributed as dist

    # pinned host copies of the inputs (one staging buffer per layer; when the
    # host cannot pin the whole cache, layers share staging buffers)
    layer_bytes = K[0].numel() * K[0].element_size() * 2
    try:
        import psutil
        avail = psutil.virtual_memory().available
    except Exception:
        avail = 64 << 30
    n_stage = max(1, min(wl.L, int(0.5 * avail // max(layer_bytes, 1))))
    hK = [K[l].cpu().pin_memory() for l in range(n_stage)]
    hV = [V[l].cpu().pin_memory() for l in range(n_stage)]
    hQ = [Q[l].cpu().pin_memory() for l in range(wl.L)]
    hX = X.cpu().pin_memory()
    hOut = [torch.empty(OUT[l].shape, dtype=OUT[l].dtype).pin_memory() for l in range(wl.L)]
    dK = [torch.empty_like(K[0]) for _ in range(2)]
    dV = [torch.empty_like(V[0]) for _ in range(2)]
    dX = torch.empty_like(X)
    dQ = [torch.empty_like(Q[0]) for _ in range(wl.L)]
    copy_stream = torch.cuda.Stream(dev)

    def e2e_step():
        dX.copy_(hX, non_blocking=True)
        for l in range(wl.L):
            dQ[l].copy_(hQ[l], non_blocking=True)
        mse = path.calibrate(dX).cpu().numpy()
        bits, _ = path.allocate(mse, w)
        path.set_bits(bits, capacity=cap)
        # double-buffered H2D of each layer's K/V on a copy stream
        done = [torch.cuda.Event() for _ in range(2)]
        free = [torch.cuda.Event() for _ in range(2)]
        for l in range(wl.L):
            s = l % 2
            with torch.cuda.stream(copy_stream):
                if l >= 2:
                    copy_stream.wait_event(free[s])
                dK[s].copy_(hK[l % n_stage], non_blocking=True)
                dV[s].copy_(hV[l % n_stage], non_blocking=True)
                done[s].record(copy_stream)
            stream.wait_event(done[s])
            path.quantize(l, dK[s], dV[s])
            free[s].record(stream)
        for l in range(wl.L):
            path.decode(l, dQ[l], OUT[l])
            hOut[l].copy_(OUT[l], non_blocking=True)
        torch.cuda.synchronize()

    e2e_step()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    steps = max(1, min(args.steps, 3))
    for _ in range(steps):
        e2e_step()
    torch.cuda.synchronize()
    el = max_over_ranks(time.perf_counter() - t0, world, dev)
    ms = el / steps * 1e3
    h2d = (hX.numel() * hX.element_size() + sum(t.numel() * t.element_size() for t in hQ)
           + wl.L * layer_bytes)
    d2h = sum(t.numel() * t.element_size() for t in hOut) + path._mse.numel() * 8
    return {"value": round(job_gbs(world, step_bytes, ms), 2), "unit": "GB/s",
            "ms_per_step": round(ms, 3), "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": steps,
            "host_staging_layers": n_stage,
            "note": "wall clock; inputs copied from pinned host memory every step"}


# --------------------------------------------------------------------------
# the CPU oracle (cpu_baseline leg and --impl reference)
# --------------------------------------------------------------------------

def oracle_sample_run(wl, tokens: int, n_calib: int, heads: int = 1, budget_s: float = 0.0):
    """Bounded sample of the workload on the CPU oracle: the calibration sweep
    of ``n_calib`` components, fit + allocation of every component, then
    quantize + pack + decode attention of (batch 0, kv head h) K+V stream
    pairs of ``tokens`` tokens, h = 0, 1, ... of layer 0, then of layer 1, ...,
    until ``heads`` pairs are done or ``budget_s`` seconds of oracle work have
    passed (input generation is not timed). Returns (algorithmic bytes,
    seconds, description)."""
    import numpy as np

    from oracle import alloc as oalloc
    from oracle import calib as ocalib
    from oracle import pipeline as opipe
    from paper_2605_06675_gb300 import synth

    S = min(tokens, wl.S)
    X = synth.calibration_sample(wl.scaled(L=1, H_kv=max(1, n_calib // 2)), device="cpu")
    signs = synth.hadamard_signs(wl.seed).numpy() if wl.hadamard else None
    xs = X.float().numpy()
    n = wl.n_components
    w = synth.importances(n, wl.sigma_lnw, wl.seed)
    allowed = list(wl.allowed)

    t0 = time.perf_counter()
    groupings = [wl.k_grouping if i % 2 == 0 else wl.v_grouping for i in range(xs.shape[0])]
    sym = [wl.v_quantizer if i % 2 else wl.k_quantizer for i in range(xs.shape[0])]
    mse = ocalib.distortion_sweep(xs, groupings, wl.hadamard, signs, symmetric=sym)
    mse_all = np.resize(mse, (n, 8))
    a, b, _ = ocalib.fit_distortion(mse_all, 2, 6, 0.96, np.arange(n) % 2)
    oalloc.allocate(w, a, b, wl.avg_bits, wl.allowed_mask)
    el = time.perf_counter() - t0
    nbytes = calib_bytes(wl, xs.shape[0], xs.shape[1])
    nblk = S // 32
    done = []
    H = max(1, wl.H_kv)
    for l in range(wl.L):
        if len(done) >= heads or (budget_s and el > budget_s):
            break
        k, v = synth.kv_layer(1, H, S, wl.dtype, wl.seed, l, wl.value_dist, "cpu")
        q = synth.queries(1, wl.H_q, wl.dtype, wl.seed, l, "cpu")
        ks, vs, qs = (t.float().numpy() for t in (k, v, q))
        for h in range(H):
            if len(done) >= heads or (budget_s and el > budget_s):
                break
            bl = np.array([[allowed[(2 * h) % len(allowed)], allowed[(2 * h + 1) % len(allowed)]]],
                          dtype=np.uint8)
            t1 = time.perf_counter()
            ol = opipe.quantize_layer(ks[:, h:h + 1], vs[:, h:h + 1], bl, wl.k_grouping,
                                      wl.v_grouping, wl.hadamard, signs,
                                      symmetric=(wl.k_quantizer, wl.v_quantizer))
            opipe.attend_layer(qs[:, h * wl.g:(h + 1) * wl.g], ol)
            el += time.perf_counter() - t1
            packed = sum(nblk * 512 * (int(x) + 1) for x in bl.reshape(-1))
            nbytes += 2 * S * 128 * 2 + packed                      # quantize: read + write
            nbytes += packed + wl.g * 128 * (2 + 4)                  # decode: packed + q + out
            done.append((l, h))
    desc = (f"oracle: calibration sweep of {xs.shape[0]} components x {xs.shape[1]} tokens, "
            f"fit + allocation of all {n} components, then quantize + pack + decode attention "
            f"of {len(done)} (batch 0, layer, kv head) K+V stream pairs of {S} tokens "
            f"(bits cycling through {allowed}); input generation not timed")
    return nbytes, el, desc


def cpu_leg_main(args, wl):
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    tokens = args.cpu_tokens or wl.S
    nbytes, el, desc = oracle_sample_run(wl, tokens, 8, heads=wl.L * wl.H_kv, budget_s=10.0)
    print(json.dumps({"value": nbytes / el / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
                      "sample": desc, "seconds": el}))


def run_cpu_leg_subprocess(wl, tokens=None):
    env = dict(os.environ)
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[var] = "1"
    env["CUDA_VISIBLE_DEVICES"] = ""
    for var in ("RANK", "WORLD_SIZE", "LOCAL_RANK", "MASTER_ADDR", "MASTER_PORT"):
        env.pop(var, None)
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--cpu-leg", "--workload", wl.name,
           "--k-quantizer", QUANTIZERS[wl.k_quantizer], "--v-quantizer", QUANTIZERS[wl.v_quantizer]]
    if tokens:
        cmd += ["--cpu-tokens", str(tokens)]
    try:
        r = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=600)
        line = [l for l in r.stdout.splitlines() if l.startswith("{")][-1]
        d = json.loads(line)
        return {"value": round(d["value"], 6), "unit": d["unit"], "cores": d["cores"],
                "kind": d["kind"], "sample": d["sample"], "seconds": round(d["seconds"], 2)}
    except Exception as e:  # report, do not fail the GPU line
        return {"value": None, "unit": "GB/s", "cores": 1, "kind": "oracle",
                "sample": f"cpu leg failed: {type(e).__name__}"}


def run_reference(args, wl, world):
    """--impl reference: the CPU oracle as it stands, bounded sample per step."""
    times = []
    tokens = min(wl.S, 8192)
    nbytes = 0
    desc = ""
    for i in range(args.warmup + args.steps):
        nbytes, el, desc = oracle_sample_run(wl, tokens, 4, heads=1)
        if i >= args.warmup:
            times.append(el)
    ms = statistics.mean(times) * 1e3
    value = nbytes / (ms * 1e-3) / 1e9
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 2),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64/f32 (numpy)",
        "data": "synthetic (seeded)", "config": {"workload": wl.name, "sample_tokens": tokens},
        "cpu_baseline": {"kind": "oracle", "cores": 1, "sample": desc, "value": round(value, 6)},
        "e2e": {"value": round(value, 6), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
        "note": "the paper ships no code; the reference arm is this repository's CPU oracle",
    }


def main():
    args = _parse()
    table, default = _workloads()
    wl = table[args.workload] if args.workload else default
    if args.layers:
        wl = wl.scaled(L=min(args.layers, wl.L))
    for kind in ("k", "v"):
        qz = getattr(args, f"{kind}_quantizer")
        if qz is not None:
            wl = wl.scaled(**{f"{kind}_quantizer": QUANTIZERS.index(qz)})
    if args.cpu_leg:
        cpu_leg_main(args, wl)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS"):
                os.environ.setdefault(var, "1")
            print(json.dumps(run_reference(args, wl, world)), flush=True)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    res = run_ours(args, wl, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
