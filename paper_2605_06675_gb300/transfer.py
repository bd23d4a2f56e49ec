"""Cross-quantizer transfer: allocate with the distortion model fitted on one
base quantizer, spend the bits on another (Sec. 3.4 "Distortion
calibration", Fig. 3; App. W "Cross-Quantizer Transfer", Table 25).

The paper's claim: each quantizer has its own beta, and an allocation made
with another quantizer's (alpha, beta) puts bits on the wrong heads. Here the
claim is exercised with the library's own calls only -- the GPU distortion
sweep of every quantizer on one calibration sample, the host fit and the
integer allocation -- and scored without a model: the weighted distortion
J = sum_i w_i D_i^B(b_i) that the allocation minimises (Eq. 1), with D^B the
sweep measured for the quantizer that holds the bits. (The paper scores with
perplexity, which needs model weights.)

Quantizer families (one calibration each; K and V are separate components,
Sec. 3.4 "K/V separation"):
  kivi      keys per channel, values per token, both min-max (the
            configurations' reading of KIVI)
  kivi_sym  keys per channel absmax ("per-channel symmetric", Sec. 2),
            values per token min-max
  rtn       keys and values per token absmax (Table 16)
  quarot    Hadamard rotation, then per token absmax (Sec. 4.1)
  turboquant Hadamard rotation, then the per-token Lloyd-Max codebook
            quantizer (App. F Table 8, App. W)
  turboquant_absmax  absmax per group with TurboQuant's group sizes
            (App. W "TurboQuant kernel"): 128 channels for keys (a whole
            row), 64 for values
The "uniform" column gives every key ceil(avg_bits) and every value
floor(avg_bits) bits (one width per kind; the same width when avg_bits is
an integer).
"""
from __future__ import annotations

import math

import numpy as np
import torch

from . import rq, synth
from .path import PackedKVPath
from .workloads import PER_CHANNEL, PER_TOKEN, PER_TOKEN_64, PER_TOKEN_128, Workload

FAMILIES = {
    "kivi": dict(k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                 k_quantizer=rq.RQ_MINMAX, v_quantizer=rq.RQ_MINMAX),
    "kivi_sym": dict(k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                     k_quantizer=rq.RQ_ABSMAX, v_quantizer=rq.RQ_MINMAX),
    "rtn": dict(k_grouping=PER_TOKEN, v_grouping=PER_TOKEN, hadamard=False,
                k_quantizer=rq.RQ_ABSMAX, v_quantizer=rq.RQ_ABSMAX),
    "quarot": dict(k_grouping=PER_TOKEN, v_grouping=PER_TOKEN, hadamard=True,
                   k_quantizer=rq.RQ_ABSMAX, v_quantizer=rq.RQ_ABSMAX),
    "turboquant": dict(k_grouping=PER_TOKEN, v_grouping=PER_TOKEN, hadamard=True,
                       k_quantizer=rq.RQ_LLOYDMAX, v_quantizer=rq.RQ_LLOYDMAX),
    "turboquant_absmax": dict(k_grouping=PER_TOKEN_128, v_grouping=PER_TOKEN_64, hadamard=False,
                              k_quantizer=rq.RQ_ABSMAX, v_quantizer=rq.RQ_ABSMAX),
}


def uniform_bits(n: int, avg_bits: float) -> np.ndarray:
    """Keys (even components) at ceil(avg_bits), values at floor(avg_bits)."""
    hi, lo = math.ceil(avg_bits), math.floor(avg_bits)
    return np.where(np.arange(n) % 2 == 0, hi, lo).astype(np.uint8)


def weighted_distortion(w: np.ndarray, mse: np.ndarray, bits: np.ndarray) -> float:
    """J = sum_i w_i D_i(b_i) with D_i(b) = mse[i][b - 1]."""
    idx = np.asarray(bits, dtype=np.int64) - 1
    return float(np.sum(np.asarray(w) * np.asarray(mse)[np.arange(len(idx)), idx]))


def transfer_matrix(wl: Workload, device="cuda", families=None, T: int = 512,
                    avg_bits: float | None = None, b_lo: int = 2, b_hi: int = 6,
                    r2_min: float = 0.96, x: torch.Tensor | None = None) -> dict:
    """Calibrate every family on the workload's calibration sample (GPU; or
    on ``x`` [n][T][128] when given), fit and allocate with each family's
    model (host), and score every allocation on every family's measured
    distortion.

    Returns dict(names, mse{f: [n][8]}, alpha{f}, beta{f}, bits{f: [n]},
    J[a][b] (allocation from family a, bits held by family b), uniform{b},
    w, avg_bits)."""
    names = list(families or FAMILIES)
    avg = wl.avg_bits if avg_bits is None else avg_bits
    if x is None:
        x = synth.calibration_sample(wl, T=T, device=device)
    n = x.shape[0]
    w = synth.importances(n, wl.sigma_lnw, wl.seed)
    classes = np.arange(n) % 2
    out = {"names": names, "mse": {}, "alpha": {}, "beta": {}, "bits": {}, "w": w,
           "avg_bits": avg}
    for f in names:
        fam = wl.scaled(**FAMILIES[f])
        signs = synth.hadamard_signs(wl.seed) if fam.hadamard else None
        path = PackedKVPath(fam, device, signs)
        mse = path.calibrate(x).cpu().numpy()
        if int(path.status.item()) != 0:
            raise RuntimeError(f"calibration of {f} reported status {int(path.status.item())}")
        alpha, beta, _ = rq.rq_fit_distortion(mse, b_lo, b_hi, r2_min, classes)
        bits, _ = rq.rq_alloc(w, alpha, beta, avg, wl.allowed_mask)
        out["mse"][f], out["alpha"][f], out["beta"][f], out["bits"][f] = mse, alpha, beta, bits
    ub = uniform_bits(n, avg)
    out["J"] = {a: {b: weighted_distortion(w, out["mse"][b], out["bits"][a]) for b in names}
                for a in names}
    out["uniform"] = {b: weighted_distortion(w, out["mse"][b], ub) for b in names}
    return out


def format_matrix(res: dict) -> str:
    """The matrix as text: rows = allocation's family, columns = quantizer,
    entries J / J(matched)."""
    names = res["names"]
    head = "alloc \\ quant".ljust(14) + "".join(n.rjust(11) for n in names)
    lines = [head]
    for a in names:
        lines.append(a.ljust(14) + "".join(
            f"{res['J'][a][b] / res['J'][b][b]:11.3f}" for b in names))
    lines.append("uniform".ljust(14) + "".join(
        f"{res['uniform'][b] / res['J'][b][b]:11.3f}" for b in names))
    lines.append("mean beta K".ljust(14) + "".join(
        f"{float(np.mean(res['beta'][b][0::2])):11.2f}" for b in names))
    lines.append("mean beta V".ljust(14) + "".join(
        f"{float(np.mean(res['beta'][b][1::2])):11.2f}" for b in names))
    lines.append("mean bits K/V".ljust(14) + "".join(
        f"{float(np.mean(res['bits'][b][0::2])):6.2f}/{float(np.mean(res['bits'][b][1::2])):4.2f}"
        for b in names))
    return "\n".join(lines)


def main(argv=None):
    import argparse
    from .workloads import ALL
    ap = argparse.ArgumentParser(description="cross-quantizer transfer matrix (weighted MSE)")
    ap.add_argument("--workload", default="qwen3_8b_L36_B16_S8192_hadamard")
    ap.add_argument("--avg-bits", type=float, default=2.5)
    ap.add_argument("--allowed", default="2,3,4,5,6,7,8")
    ap.add_argument("--tokens", type=int, default=512)
    args = ap.parse_args(argv)
    wl = {w.name: w for w in ALL}[args.workload]
    wl = wl.scaled(allowed=tuple(int(b) for b in args.allowed.split(",")))
    res = transfer_matrix(wl, torch.device("cuda", 0), T=args.tokens, avg_bits=args.avg_bits)
    print(f"{wl.name}, {res['w'].size} components, avg bits {res['avg_bits']}, "
          f"allowed {list(wl.allowed)}; J / J(matched):")
    print(format_matrix(res))


if __name__ == "__main__":
    main()
