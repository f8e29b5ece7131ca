"""Training runs of the workloads with per-step metrics as JSON lines.

The paper's compressed learning (Section 2.3, Section 4): steps of the
proximal method (the weights re-compacted to CSR after every update), then
debias steps with the pattern fixed (Section 2.4). Each step logs its phase,
the mean loss, every layer's stored count and compression rate
(stored / (rows * cols)), the step time (CUDA events on the run's stream) and
samples per second:

  python -m paper_1905_07931_gb300.run --config mlp --prox-steps 100 --debias-steps 100 --out run.jsonl
  python -m paper_1905_07931_gb300.run --config lenet --prox-steps 20 --debias-steps 20 --save lenet.npz
  python -m paper_1905_07931_gb300.run --config mlp --prox-steps 0 --load mlp.npz --debias-steps 50

Workloads: single_fc (one FC layer 784->300, upstream gradient given, prox
steps only), mlp (784-300-100-10), lenet (LeNet-5 style), fc_head
(9216-4096-4096-1000). The inputs are synthetic, drawn with the workload's
distribution (U[0,1] images, half-normal features, uniform labels) into a
pool of --batches seeded batches that the steps cycle through; each batch
is copied from pinned host memory on a copy stream while the previous step
runs (train.BatchPrefetcher).

--save writes every layer's CSR arrays (row_ptr, col_idx, val, trimmed to the
stored count) and bias to an .npz; --load puts such arrays back into the
network's buffers exactly (stored zeros included) and rebuilds the
transposed copies, so a run can resume.
"""

from __future__ import annotations

import argparse
import ctypes
import json
import sys
import time

import numpy as np
import torch

from . import csrtrain as C
from . import synth
from .train import BatchPrefetcher, SingleLayer, SparseNet, lenet_layers, mlp_layers

WORKLOADS = ("single_fc", "mlp", "lenet", "fc_head")


def _pool(config: str, cfg: dict, batches: int, seed: int):
    """A pool of input batches with the workload's distribution."""
    out = []
    for i in range(batches):
        rng = synth.rng_for(seed * 7919 + i + 1)
        if config == "mlp":
            x = synth.uniform01(rng, *cfg["X"].shape)
        elif config == "lenet":
            x = synth.uniform01(rng, *cfg["X"].shape)
        else:
            x = synth.half_normal(rng, *cfg["X"].shape)
        y = synth.labels(rng, cfg["labels"].shape[0], 10 if config in ("mlp", "lenet") else 1000)
        out.append((torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).pin_memory(),
                    torch.from_numpy(y).pin_memory()))
    return out


def build(config: str, seed: int, precision: int):
    """(net, cfg) for a workload."""
    if config == "single_fc":
        cfg = synth.single_fc(seed=seed)
        net = SingleLayer(cfg["W"], cfg["X"].shape[1], precision=precision)
        net.x.copy_(torch.from_numpy(cfg["X"]))
        net.dy.copy_(torch.from_numpy(cfg["dY"]))
        return net, cfg
    if config == "mlp":
        cfg = synth.mlp(seed=seed)
        layers, in_shape = mlp_layers(3), (cfg["X"].shape[0],)
    elif config == "lenet":
        cfg = synth.lenet(seed=seed)
        layers, in_shape = lenet_layers(), (1, 28, 28)
    elif config == "fc_head":
        cfg = synth.fc_head(seed=seed)
        layers, in_shape = mlp_layers(3), (cfg["X"].shape[0],)
    else:
        raise ValueError(f"unknown workload {config!r}")
    batch = cfg["labels"].shape[0]
    net = SparseNet(layers, cfg["W"], cfg["b"], batch, in_shape, precision=precision)
    return net, cfg


def weights(net):
    """The current CSR of every layer."""
    if isinstance(net, SingleLayer):
        return [net.W[net.cur]]
    return [net.weights(i) for i in range(len(net.params))]


def save(net, path: str):
    arrays = {}
    for i, W in enumerate(weights(net)):
        (rp, ci, v), _ = W.to_host()
        arrays[f"row_ptr{i}"], arrays[f"col_idx{i}"], arrays[f"val{i}"] = rp, ci, v
        arrays[f"shape{i}"] = np.array([W.rows, W.cols], dtype=np.int64)
        if not isinstance(net, SingleLayer):
            arrays[f"bias{i}"] = net.params[i]["b"].cpu().numpy()
    np.savez(path, **arrays)


def load(net, path: str):
    """Put saved CSR arrays (and biases) into the current buffers of net."""
    data = np.load(path)
    for i, W in enumerate(weights(net)):
        rows, cols = (int(t) for t in data[f"shape{i}"])
        if (rows, cols) != (W.rows, W.cols):
            raise ValueError(f"layer {i}: saved shape {(rows, cols)} != {(W.rows, W.cols)}")
        rp, ci, v = data[f"row_ptr{i}"], data[f"col_idx{i}"], data[f"val{i}"]
        if len(ci) > W.capacity:
            raise ValueError(f"layer {i}: {len(ci)} stored entries exceed the capacity {W.capacity}")
        W.row_ptr.copy_(torch.from_numpy(rp.astype(np.int32)))
        W.col_idx[: len(ci)].copy_(torch.from_numpy(ci.astype(np.int32)))
        W.val[: len(v)].copy_(torch.from_numpy(v.astype(np.float32)))
        ws = net.ws
        if C.validate_csr(_Plain(W) if W.transposed else W, ws) is not None:
            ws.clear_status()
            raise ValueError(f"layer {i}: the saved CSR is not valid")
        if W.transposed:
            C.csr_transpose(W, ws)
        if not isinstance(net, SingleLayer) and f"bias{i}" in data:
            net.params[i]["b"].copy_(torch.from_numpy(data[f"bias{i}"]))


class _Plain:
    """A view of a CSR without its transposed arrays (validated before they are rebuilt)."""

    def __init__(self, W):
        self._s = C.csrt_csr(W.rows, W.cols, W.capacity, C._ptr(W.row_ptr), C._ptr(W.col_idx), C._ptr(W.val),
                             None, None, None, None)

    @property
    def struct(self):
        return ctypes.byref(self._s)


def run(config: str, prox_steps: int, debias_steps: int, seed: int = 0, batches: int = 8,
        precision: int = C.CSRT_PREC_TF32, out=None, load_path: str | None = None, save_path: str | None = None):
    """Runs the phases; returns the list of per-step records (also written to
    `out`, a file object, one JSON object per line)."""
    net, cfg = build(config, seed, precision)
    if load_path:
        load(net, load_path)
    eta, lam = cfg["eta"], cfg["lambda"]
    pool = None if config == "single_fc" else _pool(config, cfg, batches, seed)
    stream = torch.cuda.current_stream()
    records = []
    phases = [("prox", prox_steps)] + ([("debias", debias_steps)] if config != "single_fc" else [])
    total = sum(c for _, c in phases)
    pf = None if pool is None else BatchPrefetcher(net)
    step = 0
    for phase, count in phases:
        for _ in range(count):
            st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            loss, lt = None, None
            st.record(stream)
            if isinstance(net, SingleLayer):
                net.step(eta, lam)
                batch = net.x.shape[1]
            else:
                # batch `step` was copied while the previous step ran; the copy
                # of the next one overlaps this step
                if step == 0:
                    pf.issue(*pool[0], after=st)
                slot = pf.acquire()
                net.set_input(pf.x[slot], pf.y[slot])   # the step reads the slot in place
                if step + 1 < total:
                    pf.issue(*pool[(step + 1) % len(pool)], after=st)
                lt = net.step(phase, eta, lam)
                pf.release(slot)
                batch = net.batch
            en.record(stream)
            torch.cuda.synchronize()
            ms = st.elapsed_time(en)
            if lt is not None:
                loss = float(lt[0].item())
            rec = {"step": step, "phase": phase, "loss": loss, "ms": round(ms, 4),
                   "samples_per_s": round(batch / (ms / 1e3), 1), "layers": []}
            for W in weights(net):
                nnz = W.nnz()
                rec["layers"].append({"rows": W.rows, "cols": W.cols, "nnz": nnz,
                                      "compression": round(nnz / max(1, W.rows * W.cols), 6)})
            flags, required = net.ws.status()
            if flags:
                rec["status"] = {"flags": flags, "required_nnz": required}
            records.append(rec)
            if out is not None:
                out.write(json.dumps(rec) + "\n")
                out.flush()
            step += 1
    if save_path:
        save(net, save_path)
    return records


def main(argv=None):
    p = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    p.add_argument("--config", choices=WORKLOADS, default="mlp")
    p.add_argument("--prox-steps", type=int, default=100)
    p.add_argument("--debias-steps", type=int, default=100)
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--batches", type=int, default=8, help="input batches in the pool the steps cycle through")
    p.add_argument("--precision", choices=["tf32", "fp32"], default="tf32")
    p.add_argument("--out", help="JSON-lines file (default: stdout)")
    p.add_argument("--save", help="write the final weights to this .npz")
    p.add_argument("--load", help="start from weights saved with --save")
    a = p.parse_args(argv)
    if not torch.cuda.is_available():
        raise SystemExit("run needs a CUDA GPU")
    prec = C.CSRT_PREC_TF32 if a.precision == "tf32" else C.CSRT_PREC_FP32
    f = open(a.out, "w") if a.out else sys.stdout
    t0 = time.perf_counter()
    try:
        recs = run(a.config, a.prox_steps, a.debias_steps, a.seed, a.batches, prec, f, a.load, a.save)
    finally:
        if a.out:
            f.close()
    print(json.dumps({"config": a.config, "steps": len(recs), "wall_s": round(time.perf_counter() - t0, 2),
                      "final_loss": recs[-1]["loss"] if recs else None,
                      "final_compression": [l["compression"] for l in recs[-1]["layers"]] if recs else None}),
          file=sys.stderr)
    return 0


if __name__ == "__main__":
    sys.exit(main())
