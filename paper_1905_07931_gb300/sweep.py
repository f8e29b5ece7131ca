"""Per-kernel timing on one sparse layer: the density / row-length / batch sweep.

The sweep takes one M x K CSR layer (default 4096 x 4096) at a density d
(1, 5, 20, 50%), with uniform (Bernoulli) or power-law (Zipf s = 1.2) row
lengths, and batch sizes n (1, 32, 256, 1024), and times each operation of the
training step on its own with CUDA events (warm-up first, inputs re-used,
L2 flushed before every timed launch):

  spmm_fwd (Y = W X), spmm_bwd_t (dX = W^T dY), weight_grad_sddmm (g at the
  stored entries), prox_update_compact twice: with the workload's lambda
  (1e-4, which makes the layer dense) and with a density-preserving lambda*
  (the (1 - d) quantile of |w - eta*G| / eta, so nnz' ~ nnz), and the dense
  weight gradient followed by the prox step, fused (weight_grad_prox_update,
  G never written) and as two calls (weight_grad_dense + prox_update_compact).

For each it prints the time, the algorithmic bytes (each operand touched
once) and the achieved GB/s, and for the products the FLOP rate and its
fraction of the GPU's FP32 FMA throughput (measured in the same run). One
operation on one shape can be selected (for profiling one kernel).

  python -m paper_1905_07931_gb300.sweep                      # the full sweep
  python -m paper_1905_07931_gb300.sweep --op prox --m 4096 --k 9216 --density 0.05 --reps 1
"""

from __future__ import annotations

import argparse
import json
import sys

import numpy as np
import torch

from . import csrtrain as C
from . import synth

DENSITIES = (0.01, 0.05, 0.20, 0.50)
BATCHES = (1, 32, 256, 1024)


def _time(fn, reps: int, flush: torch.Tensor, warmup: int = 2):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ts = []
    for i in range(reps):
        flush.fill_(float(i))
        st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        st.record()
        fn()
        en.record()
        ts.append((st, en))
    torch.cuda.synchronize()
    return float(np.median([a.elapsed_time(b) for a, b in ts]))


def density_preserving_lambda(w: np.ndarray, g: np.ndarray, eta: float, density: float) -> float:
    """lambda* = the (1 - d) quantile of |w - eta*G| / eta: keeps ~d of the entries."""
    z = np.abs(w.astype(np.float64) - eta * g.astype(np.float64)) / eta
    return float(np.quantile(z, 1.0 - density))


def run_layer(m: int, k: int, density: float, zipf: bool, batches, ops, reps: int, seed: int = 0,
              transposed: bool = True, dy_scale: float = 1.0):
    rng = synth.rng_for(seed)
    w = synth.masked_weights(rng, m, k, density, zipf=zipf)
    nmax = max(batches)
    x = synth.std_normal(rng, k, nmax)
    dy = synth.std_normal(rng, m, nmax)
    if dy_scale != 1.0:
        dy = (dy * np.float32(dy_scale)).astype(np.float32)
    g = synth.std_normal(rng, m, k)
    eta, lam = synth.ETA, synth.LAMBDA
    ws = C.Workspace(m, k, nmax)
    W = C.CSR(m, k)
    C.csr_from_dense(torch.from_numpy(w).cuda(), W, ws)
    W_out = C.CSR(m, k, transposed=transposed)
    nnz = W.nnz()
    flush = torch.empty(256 * 1024 * 1024 // 4, device="cuda")
    xd = torch.from_numpy(x).cuda()
    dyd = torch.from_numpy(dy).cuda()
    gd = torch.from_numpy(g).cuda()
    rows = []
    for n in batches:
        xn = xd[:, :n].contiguous()
        dyn = dyd[:, :n].contiguous()
        y = torch.empty(m, n, device="cuda")
        dx = torch.empty(k, n, device="cuda")
        gnz = torch.empty(max(nnz, 1), device="cuda")
        io = 4 * n * (k + m)
        spec = {
            "spmm_fwd": (lambda: C.spmm_fwd(W, xn, y, ws), 8 * nnz + 4 * (m + 1) + io, 2.0 * nnz * n),
            "spmm_bwd_t": (lambda: C.spmm_bwd_t(W, dyn, dx, ws), 8 * nnz + 4 * (k + 1) + io, 2.0 * nnz * n),
            "sddmm": (lambda: C.weight_grad_sddmm(W, dyn, xn, gnz, ws), 12 * nnz + 4 * (m + 1) + io, 2.0 * nnz * n),
        }
        for op in ("spmm_fwd", "spmm_bwd_t", "sddmm"):
            if op not in ops:
                continue
            fn, byts, flops = spec[op]
            ms = _time(fn, reps, flush)
            rows.append({"op": op, "m": m, "k": k, "density": density, "rows": "zipf" if zipf else "uniform",
                         "n": n, "nnz": nnz, "us": round(ms * 1e3, 2), "bytes": byts,
                         "gbs": round(byts / (ms / 1e3) / 1e9, 1), "tflops": round(flops / (ms / 1e3) / 1e12, 2)})
    if "fused" in ops:
        # the dense weight gradient G = dY X^T and the prox step on it: fused
        # (G never written) and as two library calls (G in HBM)
        for n in batches:
            xn = xd[:, :n].contiguous()
            dyn = dyd[:, :n].contiguous()
            g_full = torch.empty(m, k, device="cuda")
            variants = (
                ("fused", lambda: C.weight_grad_prox_update(W, dyn, xn, eta, lam, W_out, ws, g_scratch=g_full)),
                ("unfused", lambda: (C.weight_grad_dense(dyn, xn, g_full, ws, precision=C.CSRT_PREC_TF32),
                                     C.prox_update_compact(W, g_full, eta, lam, W_out, ws))),
            )
            for tag, fn in variants:
                ms = _time(fn, reps, flush)
                nnz_out = W_out.nnz()
                byts = 4 * n * (m + k) + 8 * nnz + 4 * (m + 1) + 8 * nnz_out + 4 * (m + 1)
                rows.append({"op": f"grad+prox ({tag})", "m": m, "k": k, "density": density,
                             "rows": "zipf" if zipf else "uniform", "n": n, "nnz": nnz, "nnz_out": nnz_out,
                             "us": round(ms * 1e3, 2), "bytes": byts, "gbs": round(byts / (ms / 1e3) / 1e9, 1)})
    if "prox" in ops:
        for tag, lam_v in (("lambda=1e-4", lam), ("lambda*", density_preserving_lambda(w, g, eta, density))):
            def fn(lam_v=lam_v):
                C.prox_update_compact(W, gd, eta, lam_v, W_out, ws)
            ms = _time(fn, reps, flush)
            nnz_out = W_out.nnz()
            byts = 4 * m * k + 8 * nnz + 4 * (m + 1) + 8 * nnz_out + 4 * (m + 1)
            if transposed:   # the transposed pattern: t_col, t_val, t_pos written, col and val read back
                byts += 12 * nnz_out + 8 * nnz_out + 4 * (k + 1) + 4 * (m + 1)
            rows.append({"op": f"prox ({tag})", "m": m, "k": k, "density": density,
                         "rows": "zipf" if zipf else "uniform", "n": 0, "nnz": nnz, "nnz_out": nnz_out,
                         "us": round(ms * 1e3, 2), "bytes": byts, "gbs": round(byts / (ms / 1e3) / 1e9, 1)})
    flags, _ = ws.status()
    if flags:
        raise RuntimeError(f"device status {flags}")
    return rows


def main(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--op", choices=["all", "spmm_fwd", "spmm_bwd_t", "sddmm", "prox", "fused"], default="all")
    p.add_argument("--m", type=int, default=4096)
    p.add_argument("--k", type=int, default=4096)
    p.add_argument("--density", type=float, nargs="*", default=list(DENSITIES))
    p.add_argument("--n", type=int, nargs="*", default=list(BATCHES))
    p.add_argument("--zipf", choices=["both", "yes", "no"], default="both")
    p.add_argument("--reps", type=int, default=10)
    p.add_argument("--json", action="store_true")
    p.add_argument("--dy-scale", type=float, default=1.0,
                   help="scale of dY: at eta 0.01, lambda 1e-4 and n = 256, 5e-6 keeps about a quarter of the "
                        "fused prox step's outputs, like the classifier-head step (1 keeps nearly all)")
    p.add_argument("--no-transposed", action="store_true",
                   help="prox outputs without the transposed arrays (a first layer, whose dX is not needed)")
    a = p.parse_args(argv)
    ops = {"spmm_fwd", "spmm_bwd_t", "sddmm", "prox", "fused"} if a.op == "all" else {a.op}
    zipfs = {"both": (False, True), "yes": (True,), "no": (False,)}[a.zipf]
    out = []
    for d in a.density:
        for z in zipfs:
            out += run_layer(a.m, a.k, d, z, a.n, ops, a.reps, transposed=not a.no_transposed, dy_scale=a.dy_scale)
    if ops & {"spmm_fwd", "spmm_bwd_t", "sddmm"}:
        # the CUDA-core products against the measured FP32 FMA throughput
        peak = C.fma_peak_tflops()
        for r in out:
            if "tflops" in r:
                r["fma_peak_tflops"] = round(peak, 1)
                r["fma_frac"] = round(r["tflops"] / peak, 4)
    if a.json:
        print(json.dumps(out))
    else:
        for r in out:
            extra = (f" nnz'={r['nnz_out']}" if "nnz_out" in r else
                     f" {r['tflops']:6.2f} TFLOP/s ({100 * r.get('fma_frac', 0):.1f}% of FP32 FMA)")
            print(f"{r['op']:<20s} d={r['density']:.2f} {r['rows']:<7s} n={r['n']:<5d} nnz={r['nnz']:<8d} "
                  f"{r['us']:9.1f} us {r['gbs']:8.1f} GB/s{extra}")
    return 0


if __name__ == "__main__":
    sys.exit(main())
