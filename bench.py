#!/usr/bin/env python
"""Benchmark of the RateQuant packed mixed-bit KV path on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
  a1  distortion sweep b = 1..8 on the calibration sample (GPU)
  a2  fit D(b) = alpha beta^-b (host), a3 integer allocation (host) + layout
  a4/a5  quantize + bit-pack every layer of the cache (GPU, one launch/layer)
  a6/a7  split-K decode attention on the packed cache for every layer (GPU)

Prints ONE JSON line (rank 0). ``value`` is the metric's first term, the
decode-attention GB/s (decode bytes of all layers over the decode time of a
step); quantize-pack, calibration and the other large configurations are
under ``components``. ``--impl reference`` times the CPU oracle (the only
reference that exists: the paper ships no code) on the host cores.
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
    ap.add_argument("--configs", default=None,
                    help="comma-separated further workloads measured in the same run under "
                         "components.configs (default with the default workload: the Qwen3 "
                         "and 70B-shaped caches; 'none' to skip)")
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


def _local_includes(path: str) -> list:
    """The files a C/CUDA source includes with #include "...", found next to
    it or in include/, recursively (each once, in first-seen order)."""
    import re
    csrc = os.path.join(ROOT, "paper_2605_06675_gb300", "csrc")
    seen, order, todo = set(), [], [path]
    while todo:
        p = todo.pop(0)
        if p in seen:
            continue
        seen.add(p)
        order.append(p)
        for inc in re.findall(r'^\s*#\s*include\s+"([^"]+)"', open(p, encoding="utf-8").read(), re.M):
            for d in (os.path.dirname(p), csrc, os.path.join(ROOT, "include")):
                cand = os.path.join(d, inc)
                if os.path.exists(cand):
                    todo.append(cand)
                    break
    return order


def kernel_source_hash(name: str) -> str:
    """sha256[:16] of a kernel's translation unit together with every local
    header it includes (recursively), comments stripped: a record goes stale
    when the code the kernel is compiled from changes, not when a comment or
    an unrelated header does."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_2605_06675_gb300", "csrc")
    h = hashlib.sha256()
    for path in _local_includes(os.path.join(csrc, name)):
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

EXTRA_CONFIGS = ["qwen3_8b_L36_B16_S8192_hadamard", "llama70b_L80_B1_S131072_kivi"]


class Arm:
    """One workload on the device: inputs resident in HBM, the library path,
    and the step (calibrate -> fit + allocate -> quantize every layer ->
    decode every layer), the two per-layer loops replayed as CUDA graphs."""

    def __init__(self, wl, dev, stream, use_graphs):
        import torch
        from paper_2605_06675_gb300 import synth
        from paper_2605_06675_gb300.path import PackedKVPath
        self.wl, self.dev, self.stream = wl, dev, stream
        signs = synth.hadamard_signs(wl.seed) if wl.hadamard else None
        self.K, self.V, self.Q, self.OUT = [], [], [], []
        for l in range(wl.L):
            k, v = synth.kv_layer(wl.B, wl.H_kv, wl.S, wl.dtype, wl.seed, l, wl.value_dist, dev)
            self.K.append(k)
            self.V.append(v)
            self.Q.append(synth.queries(wl.B, wl.H_q, wl.dtype, wl.seed, l, dev))
            self.OUT.append(torch.empty((wl.B, wl.H_q, 128), dtype=torch.float32, device=dev))
        self.X = synth.calibration_sample(wl, device=dev)
        self.n, self.T = self.X.shape[0], self.X.shape[1]
        self.w = synth.importances(self.n, wl.sigma_lnw, wl.seed)
        self.path = PackedKVPath(wl, dev, signs)
        # capacity of the packed cache: every stream at the widest allowed width
        self.cap = wl.L * wl.B * wl.H_kv * 2 * (wl.S // 32) * 512 * (max(wl.allowed) + 1)
        mse0 = self.path.calibrate(self.X).cpu().numpy()
        bits0, _ = self.path.allocate(mse0, self.w)
        self.path.set_bits(bits0, capacity=self.cap)
        self.path.decode_workspace()
        torch.cuda.synchronize()
        self.graphs = None
        self.use_graphs = use_graphs
        self.launch_mode = "per-layer launches"

    def step(self, ev=None, host_ms=None):
        import time as _t
        p, wl, st = self.path, self.wl, self.stream
        if ev is not None:
            ev[0].record(st)
        mse = p.calibrate(self.X)
        if ev is not None:
            ev[1].record(st)
        mse_h = mse.cpu().numpy()                       # D2H, synchronises
        t0 = _t.perf_counter()
        bits, _ = p.allocate(mse_h, self.w)
        p.set_bits(bits, capacity=self.cap)
        if host_ms is not None:
            host_ms.append((_t.perf_counter() - t0) * 1e3)
        if ev is not None:
            ev[2].record(st)
        if self.graphs is not None:
            self.graphs[0].replay()
        else:
            for l in range(wl.L):
                p.quantize(l, self.K[l], self.V[l])
        if ev is not None:
            ev[3].record(st)
        if self.graphs is not None:
            self.graphs[1].replay()
        else:
            for l in range(wl.L):
                p.decode(l, self.Q[l], self.OUT[l])
        if ev is not None:
            ev[4].record(st)
        return bits

    def capture(self):
        """The quantize and decode loops of a step as two CUDA graphs (the
        kernels read the widths and offsets set_bits writes in place)."""
        import torch
        if not self.use_graphs:
            return
        try:
            gq, gd = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
            with torch.cuda.graph(gq, stream=self.stream):
                for l in range(self.wl.L):
                    self.path.quantize(l, self.K[l], self.V[l])
            with torch.cuda.graph(gd, stream=self.stream):
                for l in range(self.wl.L):
                    self.path.decode(l, self.Q[l], self.OUT[l])
            self.graphs = (gq, gd)
            self.launch_mode = "cuda graphs (quantize loop, decode loop)"
            self.step()
            torch.cuda.synchronize()
        except RuntimeError as e:
            self.graphs = None
            self.launch_mode = f"per-layer launches (graph capture failed: {str(e)[:80]})"
            torch.cuda.synchronize()

    def timed(self, steps, world, clocks=None):
        """Time exactly `steps` steps (CUDA events on the launching stream);
        returns the per-phase means and the max-over-ranks step time."""
        import torch
        import torch.distributed as dist
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(steps)]
        host_ms = []
        if clocks is not None:
            clocks.start()
            time.sleep(0.15)
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        start.record(self.stream)
        bits = None
        for i in range(steps):
            bits = self.step(evs[i], host_ms)
        end.record(self.stream)
        torch.cuda.synchronize()
        clk = clocks.stop() if clocks is not None else None
        total_ms = max_over_ranks(start.elapsed_time(end), world, self.dev)
        if world > 1:
            dist.barrier()
        r = {
            "calib_ms": statistics.mean(e[0].elapsed_time(e[1]) for e in evs),
            "quant_ms": max_over_ranks(statistics.mean(e[2].elapsed_time(e[3]) for e in evs), world, self.dev),
            "dec_ms": max_over_ranks(statistics.mean(e[3].elapsed_time(e[4]) for e in evs), world, self.dev),
            "host_ms": statistics.mean(host_ms), "ms_step": total_ms / steps, "clocks": clk,
            "bits": bits, "steps": steps,
        }
        wl = self.wl
        r["qb"] = sum(quant_bytes_layer(wl, bits[l]) for l in range(wl.L))
        r["db"] = sum(decode_bytes_layer(wl, bits[l]) for l in range(wl.L))
        r["cb"] = calib_bytes(wl, self.n, self.T)
        return r


def summary(wl, r, peak, world):
    """Per-workload numbers of the metric: decode-attention GB/s (fraction of
    the measured HBM peak and of 8 TB/s), tokens/s, quantize GB/s."""
    d_gbs = job_gbs(world, r["db"], r["dec_ms"])
    q_gbs = job_gbs(world, r["qb"], r["quant_ms"])
    return {
        "workload": wl.name,
        "decode_attention": {"gbs": round(d_gbs, 1), "frac_of_measured_hbm": round(d_gbs / peak, 4),
                             "frac_of_8TBs": round(d_gbs / 8000.0, 4),
                             "tokens_per_s": round(world * wl.B / (r["dec_ms"] * 1e-3), 1),
                             "us_per_layer": round(r["dec_ms"] * 1e3 / wl.L, 2),
                             "ms_per_step": round(r["dec_ms"], 4), "bytes_per_step": int(r["db"])},
        "quantize_pack": {"gbs": round(q_gbs, 1), "frac_of_measured_hbm": round(q_gbs / peak, 4),
                          "frac_of_8TBs": round(q_gbs / 8000.0, 4),
                          "us_per_layer": round(r["quant_ms"] * 1e3 / wl.L, 2),
                          "ms_per_step": round(r["quant_ms"], 4), "bytes_per_step": int(r["qb"])},
        "calibrate": {"ms_per_step": round(r["calib_ms"], 4)},
        "fit_alloc_layout_host": {"ms_per_step": round(r["host_ms"], 4)},
        "ms_per_step": round(r["ms_step"], 4), "steps": r["steps"],
        "avg_bits_allocated": round(float(r["bits"].mean()), 4),
    }


def roofline_of(kernel, per_launch_bytes, per_launch_ms, peak, peak_kind, traffic):
    achieved = per_launch_bytes / (per_launch_ms * 1e-3) / 1e9
    return {"bound": "hbm", "kernel": kernel, "achieved": round(achieved, 1), "peak": peak,
            "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": traffic,
            "algorithmic_bytes_per_launch": int(per_launch_bytes),
            "peak_source": f"{peak_kind} hbm_gbs"}


def run_ours(args, wl, rank, world, local_rank):
    import torch

    from paper_2605_06675_gb300 import build as _b

    if not os.path.exists(_b.LIB):
        if rank == 0:
            _b.build()
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    # a stream of our own: the per-layer loops are captured as CUDA graphs on it
    stream = torch.cuda.Stream(dev)
    torch.cuda.set_stream(stream)
    peak, peak_kind = _peaks()

    arm = Arm(wl, dev, stream, not args.no_graphs)
    for _ in range(args.warmup):
        arm.step()
    torch.cuda.synchronize()
    arm.capture()
    r = arm.timed(args.steps, world, ClockSampler(local_rank))
    main = summary(wl, r, peak, world)

    # the metric's first term over the whole job: decode-attention bytes of
    # every rank / the slowest rank's decode time per step
    value = job_gbs(world, r["db"], r["dec_ms"])
    # dominant kernel of the step by time share (per launch = one layer)
    shares = {"quantize_pack": r["quant_ms"], "decode_attention": r["dec_ms"], "calibrate": r["calib_ms"]}
    dom = max(shares, key=shares.get)
    rq_ = roofline_of("quantize_pack", r["qb"] / wl.L, r["quant_ms"] / wl.L, peak, peak_kind,
                      recorded_traffic("quantize_pack", wl.name))
    rd_ = roofline_of("decode_attention (split + merge)", r["db"] / wl.L, r["dec_ms"] / wl.L, peak,
                      peak_kind, recorded_traffic("decode_split", wl.name))
    roofline = rq_ if dom == "quantize_pack" else rd_

    result = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(r["ms_step"], 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16 in; f32 quantizer; f16 x f16 -> f32 mma attention",
        "data": "synthetic (seeded; Llama-3/Qwen3-shaped KV caches, random q)",
        "config": {"workload": wl.name, "L": wl.L, "B": wl.B, "H_kv": wl.H_kv, "H_q": wl.H_q,
                   "S": wl.S, "head_dim": 128, "group": 32, "bits_allowed": list(wl.allowed),
                   "avg_bits": wl.avg_bits, "k_grouping": "per_channel" if wl.k_grouping else "per_token",
                   "v_grouping": "per_channel" if wl.v_grouping else "per_token",
                   "hadamard": wl.hadamard, "k_quantizer": QUANTIZERS[wl.k_quantizer],
                   "v_quantizer": QUANTIZERS[wl.v_quantizer],
                   "calib_tokens": arm.T, "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (no flush)", "launch": arm.launch_mode},
        "value_is": "decode-attention GB/s: decode bytes (packed codes + scale/zero + q + fp32 out) "
                    "of all layers / decode time per step, over all ranks",
        "components": dict(main, configs={}),
        "roofline": roofline,
        "roofline_decode": rd_,
        "clocks": r["clocks"],
        "gpu_launches": args.steps * (2 + 3 * wl.L),
    }

    if not args.no_e2e:
        result["e2e"] = run_e2e(args, arm, world, r)
    del arm
    torch.cuda.synchronize()
    torch.cuda.empty_cache()

    # the other large configurations, measured the same way in the same run
    extra = [] if (args.configs or "") == "none" else (
        args.configs.split(",") if args.configs else (EXTRA_CONFIGS if args.workload is None and not args.layers else []))
    table, _ = _workloads()
    for name in extra:
        if name == wl.name or name not in table:
            continue
        xwl = table[name]
        xarm = Arm(xwl, dev, stream, not args.no_graphs)
        xw = min(args.warmup, 3) if args.warmup >= 3 else 3
        for _ in range(xw):
            xarm.step()
        torch.cuda.synchronize()
        xarm.capture()
        xr = xarm.timed(max(3, min(args.steps, 10)), world)
        s = summary(xwl, xr, peak, world)
        s["warmup"] = xw
        s["roofline_decode"] = roofline_of("decode_attention (split + merge)", xr["db"] / xwl.L,
                                           xr["dec_ms"] / xwl.L, peak, peak_kind,
                                           recorded_traffic("decode_split", xwl.name))
        s["roofline_quantize"] = roofline_of("quantize_pack", xr["qb"] / xwl.L, xr["quant_ms"] / xwl.L,
                                             peak, peak_kind, recorded_traffic("quantize_pack", xwl.name))
        result["components"]["configs"][name] = s
        del xarm
        torch.cuda.synchronize()
        torch.cuda.empty_cache()

    if rank == 0 and not args.no_cpu_baseline and world == 1:
        result["cpu_baseline"] = run_cpu_leg_subprocess(wl)
    return result


def run_e2e(args, arm, world, r):
    """The step through the public API with HOST inputs: every step moves the
    calibration sample, each layer's K/V and q from pinned host memory to the
    device and reads every layer's output back. The calibration sample and q
    are copied; K and V are read by the quantize kernel straight from the
    pinned host buffers (rq_quantize_pack accepts device-addressable host
    memory), which on GB300's NVLink-C2C moves them at about twice the rate of
    copy-engine transfers of the same buffers. The value is the metric's
    decode-attention bytes over that whole step's time (host transfers
    included); the step's algorithmic bytes over the same time are under
    step_gbs."""
    import torch
    import torch.distributed as dist

    wl, path, dev, stream = arm.wl, arm.path, arm.dev, arm.stream
    K, V, Q, OUT, X = arm.K, arm.V, arm.Q, arm.OUT, arm.X
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
    dX = torch.empty_like(X)
    dQ = [torch.empty_like(Q[0]) for _ in range(wl.L)]

    def e2e_step():
        dX.copy_(hX, non_blocking=True)
        for l in range(wl.L):
            dQ[l].copy_(hQ[l], non_blocking=True)
        mse = path.calibrate(dX).cpu().numpy()
        bits, _ = path.allocate(mse, arm.w)
        path.set_bits(bits, capacity=arm.cap)
        # each layer's K/V read by the quantize kernel from pinned host memory
        for l in range(wl.L):
            path.quantize(l, hK[l % n_stage], hV[l % n_stage])
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
    step_bytes = r["qb"] + r["db"] + r["cb"]
    return {"value": round(job_gbs(world, r["db"], ms), 3), "unit": "GB/s",
            "ms_per_step": round(ms, 3), "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": steps,
            "step_gbs": round(job_gbs(world, step_bytes, ms), 2),
            "host_staging_layers": n_stage,
            "note": "wall clock of the whole step through the public calls; inputs moved from "
                    "pinned host memory every step (calibration sample and q copied, K/V read in "
                    "place by the quantize kernel over the host link) and outputs read back; value "
                    "= decode-attention bytes / that time"}


# --------------------------------------------------------------------------
# the CPU oracle (cpu_baseline leg and --impl reference)
# --------------------------------------------------------------------------

def _oracle_task(t):
    """One (layer, kv head) K+V stream pair of batch 0 through the oracle:
    quantize + pack, then decode attention on the dequantized cache (inputs
    drawn by synth, not timed). Returns bytes and seconds of both phases."""
    name, layer, head, tokens = t
    import numpy as np

    from oracle import pipeline as opipe
    from paper_2605_06675_gb300 import synth
    from paper_2605_06675_gb300 import workloads as W
    wl = {w.name: w for w in W.ALL}[name]
    S = min(tokens, wl.S)
    k, v = synth.kv_layer(1, 1, S, wl.dtype, wl.seed + 7 * head, layer, wl.value_dist, "cpu")
    q = synth.queries(1, wl.g, wl.dtype, wl.seed + 7 * head, layer, "cpu")
    signs = synth.hadamard_signs(wl.seed).numpy() if wl.hadamard else None
    allowed = list(wl.allowed)
    bl = np.array([[allowed[(2 * head) % len(allowed)], allowed[(2 * head + 1) % len(allowed)]]],
                  dtype=np.uint8)
    ks, vs, qs = (x.float().numpy() for x in (k, v, q))
    t0 = time.perf_counter()
    ol = opipe.quantize_layer(ks, vs, bl, wl.k_grouping, wl.v_grouping, wl.hadamard, signs,
                              symmetric=(wl.k_quantizer, wl.v_quantizer))
    t1 = time.perf_counter()
    opipe.attend_layer(qs, ol)
    t2 = time.perf_counter()
    packed = sum((S // 32) * 512 * (int(b) + 1) for b in bl.reshape(-1))
    return {"qbytes": 2 * S * 128 * 2 + packed, "qsec": t1 - t0,
            "dbytes": packed + wl.g * 128 * (2 + 4), "dsec": t2 - t1}


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


class OraclePool:
    """A pool of `cores` oracle processes (spawned, one thread each)."""

    def __init__(self, cores):
        import multiprocessing as mp
        for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
            os.environ[var] = "1"
        self.cores = cores
        self.pool = mp.get_context("spawn").Pool(cores)

    def run(self, tasks):
        """Rates of one batch of tasks run in parallel: per-phase task times
        scaled by the pool's measured speedup (sum of task times / wall)."""
        t0 = time.perf_counter()
        res = self.pool.map(_oracle_task, tasks, chunksize=1)
        wall = time.perf_counter() - t0
        busy = sum(x["qsec"] + x["dsec"] for x in res)
        speedup = busy / wall if wall > 0 else 1.0
        qb, qs = sum(x["qbytes"] for x in res), sum(x["qsec"] for x in res)
        db, ds = sum(x["dbytes"] for x in res), sum(x["dsec"] for x in res)
        return {"decode_gbs": db / (ds / speedup) / 1e9, "quantize_gbs": qb / (qs / speedup) / 1e9,
                "wall_s": wall, "speedup": speedup, "tasks": len(tasks)}

    def close(self):
        self.pool.close()
        self.pool.join()


def oracle_tasks(wl, n, tokens, start=0):
    """n (layer, kv head) stream pairs of batch 0, layer-major from `start`."""
    return [(wl.name, (start + i) // wl.H_kv % wl.L, (start + i) % wl.H_kv, tokens) for i in range(n)]


def cpu_leg_main(args, wl):
    """The oracle on the host cores: all cores (a spawned pool, one stream
    pair per task) and one core (the same tasks in this process)."""
    tokens = args.cpu_tokens or wl.S
    cores = host_cores()
    t_start = time.perf_counter()
    pool = OraclePool(cores)
    pool.run(oracle_tasks(wl, cores, min(tokens, 1024)))          # start-up (imports), not reported
    all_cores = pool.run(oracle_tasks(wl, 2 * cores, tokens))
    pool.close()
    one = [_oracle_task(t) for t in oracle_tasks(wl, 3, tokens)]
    d1 = sum(x["dbytes"] for x in one) / sum(x["dsec"] for x in one) / 1e9
    q1 = sum(x["qbytes"] for x in one) / sum(x["qsec"] for x in one) / 1e9
    S = min(tokens, wl.S)
    # a whole step of the workload (every layer, batch row and kv head at the
    # workload's average width) at the sample's all-core rates: extrapolated
    streams = wl.L * wl.B * wl.H_kv * 2
    packed = streams * (wl.S // 32) * 512 * (wl.avg_bits + 1)
    q_full = streams * wl.S * 128 * 2 + packed
    d_full = packed + wl.L * wl.B * wl.H_q * 128 * (2 + 4)
    full_step_s = q_full / (all_cores["quantize_gbs"] * 1e9) + d_full / (all_cores["decode_gbs"] * 1e9)
    sample = (f"oracle (numpy, fp64 softmax) on {2 * cores} (layer, kv head) K+V stream pairs of batch 0, "
              f"{S} tokens each, widths cycling through {list(wl.allowed)}, spread over {cores} "
              f"processes; then 3 pairs on one core; input generation not timed")
    print(json.dumps({
        "value": all_cores["decode_gbs"], "unit": "GB/s", "cores": cores, "kind": "oracle",
        "sample": sample, "quantize_gbs": all_cores["quantize_gbs"],
        "pool_speedup": all_cores["speedup"], "pool_wall_s": all_cores["wall_s"],
        "single_core": {"value": d1, "quantize_gbs": q1, "cores": 1},
        "seconds": time.perf_counter() - t_start,
        "extrapolated_full_step_s": full_step_s,
        "extrapolated_note": "quantize + decode of every stream of the workload at the sample's "
                             "all-core rates (not run)"}))


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
        r = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=900)
        line = [l for l in r.stdout.splitlines() if l.startswith("{")][-1]
        d = json.loads(line)
        for key in ("value", "quantize_gbs"):
            d[key] = round(d[key], 6)
        d["single_core"] = {k: (round(v, 6) if isinstance(v, float) else v)
                            for k, v in d["single_core"].items()}
        d["seconds"] = round(d["seconds"], 2)
        return d
    except Exception as e:  # report, do not fail the GPU line
        return {"value": None, "unit": "GB/s", "cores": host_cores(), "kind": "oracle",
                "sample": f"cpu leg failed: {type(e).__name__}"}


def run_reference(args, wl, world):
    """--impl reference: the CPU oracle as it stands on the host cores, on the
    same workload, metric and unit as our arm: each step one stream pair per
    core at the workload's full sequence length."""
    cores = host_cores()
    pool = OraclePool(cores)
    tokens = wl.S
    pool.run(oracle_tasks(wl, cores, min(tokens, 1024)))          # start-up, not timed
    rates, qrates, walls = [], [], []
    for i in range(args.warmup + args.steps):
        r = pool.run(oracle_tasks(wl, cores, tokens, start=i * cores))
        if i >= args.warmup:
            rates.append(r["decode_gbs"])
            qrates.append(r["quantize_gbs"])
            walls.append(r["wall_s"])
    pool.close()
    value = statistics.mean(rates)
    desc = (f"oracle (numpy) on {cores} host processes, each step {cores} (layer, kv head) K+V "
            f"stream pairs of batch 0 at {tokens} tokens (quantize + pack, then decode attention); "
            "rate = decode-attention bytes / the decode phase's share of the pool's wall time")
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(walls) * 1e3, 2),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64/f32 (numpy)",
        "data": "synthetic (seeded)", "config": {"workload": wl.name, "sample_tokens": tokens},
        "cpu_baseline": {"kind": "oracle", "cores": cores, "sample": desc, "value": round(value, 6),
                         "quantize_gbs": round(statistics.mean(qrates), 6)},
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
