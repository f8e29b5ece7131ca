"""LeNet-5 inference with compressed (CSR) weights against the dense network.

The paper's inference comparison (Section 4.5, the table of inference speedups
on LeNet-5 / MNIST) runs the same network once with its compressed weights and
sparse kernels and once with the full dense weights, and reports the speedup
(2x on a GTX 1080 Ti, 1.2x on a Mali-T860). This module restates it on one
GPU:

  network   LeNet-5 of Section 4: conv 5x5x20, max-pool 2, conv 5x5x50,
            max-pool 2, fc 800->500 + ReLU, fc 500->10 (Caffe flatten order).
  weights   He-normal values on uniform random patterns with the stored
            counts the paper reports for SpC in its LeNet-5 layer table
            (conv1 158/500, conv2 2101/25,000, fc1 10,804/400,000,
            fc2 270/5,000); the dense network holds the same values with
            zeros elsewhere (so both compute the same function).
  inputs    synthetic MNIST-shaped images, U[0, 1] 28 x 28, 10,000 of them
            (the size of the MNIST test set), forwarded in batches.
  paths     compressed: csrt_conv2d_sparse_fwd for both convolutions (the
            input is read in place, never unfolded), max-pool, flatten,
            spmm_fwd_bias_act for both fully connected layers.
            dense GEMM: the Caffe lowering the paper's dense reference uses,
            csrt_im2col + cuBLAS SGEMM (float32, TF32 off) for the
            convolutions, the same glue kernels, cuBLAS SGEMM for the fully
            connected layers.
            dense cuDNN: torch conv2d / linear (cuDNN and cuBLAS, float32,
            TF32 off), a stronger dense baseline than the lowering.

Each path's forward of one batch is captured in a CUDA graph; the timed
region replays it for every batch of the 10,000 images, with CUDA events on
the replay stream, after warm-up; the L2 is flushed before each timed pass.
Before timing, the three paths' logits on the first batch are checked
against each other (the tests check them against the CPU oracle).

  python -m paper_1905_07931_gb300.infer                 # batch 1000
  python -m paper_1905_07931_gb300.infer --batch 128 --json
"""

from __future__ import annotations

import argparse
import json
import sys

import numpy as np
import torch

from . import csrtrain as C
from . import synth

# stored / total weights per layer: SpC column of the paper's LeNet-5 layer table
SPC_NNZ = (158, 2101, 10804, 270)
SHAPES = ((20, 25), (50, 500), (500, 800), (10, 500))     # (M, K) of conv1, conv2, fc1, fc2
PAPER = {"gtx1080ti_ms": {"compressed": 8572, "dense": 16977, "speedup": 2.0},
         "mali_t860_ms": {"compressed": 506067, "dense": 606699, "speedup": 1.2},
         "model_size": {"compressed": "148KB", "dense": "5.0MB"}}


def lenet_weights(seed: int = 0):
    """Dense M x K weights with exactly SPC_NNZ stored entries each, and biases."""
    rng = synth.rng_for(seed)
    ws, bs = [], []
    for (m, k), nnz in zip(SHAPES, SPC_NNZ):
        w = np.zeros(m * k, dtype=np.float32)
        pos = rng.choice(m * k, size=nnz, replace=False)
        vals = rng.standard_normal(nnz) * np.sqrt(2.0 / k)
        vals[vals == 0] = 1e-3
        w[pos] = vals.astype(np.float32)
        ws.append(w.reshape(m, k))
        bs.append((rng.standard_normal(m) * 0.01).astype(np.float32))
    return ws, bs


class Compressed:
    """The CSR network: sparse convolutions read the input in place."""

    def __init__(self, ws, bs, batch: int):
        B = batch
        self.B = B
        self.ws_ = C.Workspace(500, 800, max(B * 576, 1))
        self.W = []
        for w in ws:
            csr = C.CSR(*w.shape, transposed=False)
            C.csr_from_dense(torch.from_numpy(w).cuda(), csr, self.ws_)
            self.W.append(csr)
        self.b = [torch.from_numpy(b).cuda() for b in bs]
        f = dict(device="cuda", dtype=torch.float32)
        self.x = torch.zeros(1, B * 784, **f)
        self.c1 = torch.zeros(20, B * 576, **f)
        self.p1 = torch.zeros(20, B * 144, **f)
        self.i1 = torch.zeros(20 * B * 144, dtype=torch.int8, device="cuda")
        self.c2 = torch.zeros(50, B * 64, **f)
        self.p2 = torch.zeros(50, B * 16, **f)
        self.i2 = torch.zeros(50 * B * 16, dtype=torch.int8, device="cuda")
        self.fl = torch.zeros(800, B, **f)
        self.h = torch.zeros(500, B, **f)
        self.logits = torch.zeros(10, B, **f)

    def forward(self, s=None):
        B = self.B
        C.conv2d_sparse_fwd(self.W[0], self.x, 1, B, 28, 28, 5, self.b[0], False, self.c1, s)
        C.maxpool2_fwd(self.c1, 20, B, 24, 24, self.p1, self.i1, s)
        C.conv2d_sparse_fwd(self.W[1], self.p1, 20, B, 12, 12, 5, self.b[1], False, self.c2, s)
        C.maxpool2_fwd(self.c2, 50, B, 8, 8, self.p2, self.i2, s)
        C.flatten(self.p2, 50, B, 16, self.fl, s)
        C.spmm_fwd_bias_act(self.W[2], self.fl, self.b[2], True, self.h, self.ws_, s)
        C.spmm_fwd_bias_act(self.W[3], self.h, self.b[3], False, self.logits, self.ws_, s)


class DenseGemm:
    """The dense network lowered as in Caffe: im2col + SGEMM."""

    def __init__(self, ws, bs, batch: int):
        B = self.B = batch
        self.W = [torch.from_numpy(w).cuda() for w in ws]
        self.b = [torch.from_numpy(b).cuda() for b in bs]
        f = dict(device="cuda", dtype=torch.float32)
        self.x = torch.zeros(1, B * 784, **f)
        self.cols1 = torch.zeros(25, B * 576, **f)
        self.c1 = torch.zeros(20, B * 576, **f)
        self.p1 = torch.zeros(20, B * 144, **f)
        self.i1 = torch.zeros(20 * B * 144, dtype=torch.int8, device="cuda")
        self.cols2 = torch.zeros(500, B * 64, **f)
        self.c2 = torch.zeros(50, B * 64, **f)
        self.p2 = torch.zeros(50, B * 16, **f)
        self.i2 = torch.zeros(50 * B * 16, dtype=torch.int8, device="cuda")
        self.fl = torch.zeros(800, B, **f)
        self.h = torch.zeros(500, B, **f)
        self.logits = torch.zeros(10, B, **f)

    def forward(self, s=None):
        B = self.B
        C.im2col(self.x, 1, B, 28, 28, 5, self.cols1, s)
        torch.mm(self.W[0], self.cols1, out=self.c1)
        C.bias_act_fwd(self.c1, self.b[0], False, s)
        C.maxpool2_fwd(self.c1, 20, B, 24, 24, self.p1, self.i1, s)
        C.im2col(self.p1, 20, B, 12, 12, 5, self.cols2, s)
        torch.mm(self.W[1], self.cols2, out=self.c2)
        C.bias_act_fwd(self.c2, self.b[1], False, s)
        C.maxpool2_fwd(self.c2, 50, B, 8, 8, self.p2, self.i2, s)
        C.flatten(self.p2, 50, B, 16, self.fl, s)
        torch.mm(self.W[2], self.fl, out=self.h)
        C.bias_act_fwd(self.h, self.b[2], True, s)
        torch.mm(self.W[3], self.h, out=self.logits)
        C.bias_act_fwd(self.logits, self.b[3], False, s)


class DenseCudnn:
    """The dense network through cuDNN convolutions (NCHW, batch-major)."""

    def __init__(self, ws, bs, batch: int):
        self.B = batch
        self.w1 = torch.from_numpy(ws[0].reshape(20, 1, 5, 5)).cuda()
        self.w2 = torch.from_numpy(ws[1].reshape(50, 20, 5, 5)).cuda()
        self.w3 = torch.from_numpy(ws[2]).cuda()
        self.w4 = torch.from_numpy(ws[3]).cuda()
        self.b = [torch.from_numpy(b).cuda() for b in bs]
        self.x = torch.zeros(batch, 1, 28, 28, device="cuda")
        self.logits = None

    def forward(self, s=None):
        F = torch.nn.functional
        y = F.max_pool2d(F.conv2d(self.x, self.w1, self.b[0]), 2)
        y = F.max_pool2d(F.conv2d(y, self.w2, self.b[1]), 2)
        y = F.relu(F.linear(y.reshape(self.B, 800), self.w3, self.b[2]))
        self.logits = F.linear(y, self.w4, self.b[3])


def _load(path, imgs):
    """Copy a batch (B, 28, 28) into the path's input in its layout."""
    if isinstance(path, DenseCudnn):
        path.x.copy_(imgs.reshape(path.B, 1, 28, 28))
    else:
        path.x.copy_(imgs.reshape(1, -1))


def _logits_bm(path):
    """Logits as (B, 10)."""
    return path.logits if isinstance(path, DenseCudnn) else path.logits.t()


def logits_of(path, images: np.ndarray) -> np.ndarray:
    """(B, 10) logits of one batch through `path`."""
    _load(path, torch.from_numpy(np.ascontiguousarray(images)).cuda())
    path.forward()
    torch.cuda.synchronize()
    return _logits_bm(path).cpu().numpy().astype(np.float64)


def cross_check(paths, images: np.ndarray, rtol=1e-4, rtol_cudnn=5e-3):
    """Max difference of each path's logits from the compressed path's, relative
    to the largest logit (the three compute the same function). cuDNN picks
    its convolution algorithm by shape (at large batches a transform-based
    one that rounds differently), hence its looser bound."""
    ref = logits_of(paths["compressed"], images)
    scale = np.abs(ref).max() + 1e-30
    out = {}
    for name, p in paths.items():
        err = float(np.abs(logits_of(p, images) - ref).max() / scale)
        if not err <= (rtol_cudnn if name == "dense_cudnn" else rtol):
            raise AssertionError(f"{name} logits differ from the compressed network's: {err:.3g}")
        out[name] = err
    return out


def time_paths(paths, images: torch.Tensor, batch: int, reps: int, warmup: int = 3):
    """ms per pass over all images (batches of `batch`), per path, from CUDA events around graph replays."""
    n_batches = images.shape[0] // batch
    flush = torch.empty(256 * 1024 * 1024 // 4, device="cuda")
    res = {}
    prev_tf32 = torch.backends.cuda.matmul.allow_tf32, torch.backends.cudnn.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.backends.cudnn.allow_tf32 = False
    try:
        for name, p in paths.items():
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(s):
                _load(p, images[:batch])
                for _ in range(warmup):
                    p.forward(s)
                torch.cuda.synchronize()
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=s):
                    p.forward(s)
                torch.cuda.synchronize()
                times = []
                for r in range(reps + warmup):
                    flush.fill_(float(r))
                    st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    total = 0.0
                    for bi in range(n_batches):
                        _load(p, images[bi * batch:(bi + 1) * batch])
                        st.record(s)
                        g.replay()
                        en.record(s)
                        en.synchronize()
                        total += st.elapsed_time(en)
                    if r >= warmup:
                        times.append(total)
            torch.cuda.current_stream().wait_stream(s)
            res[name] = float(np.median(times))
    finally:
        torch.backends.cuda.matmul.allow_tf32, torch.backends.cudnn.allow_tf32 = prev_tf32
    return res


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--batch", type=int, default=1000)
    ap.add_argument("--images", type=int, default=10000)
    ap.add_argument("--reps", type=int, default=5)
    ap.add_argument("--json", action="store_true")
    a = ap.parse_args(argv)
    if a.images % a.batch:
        raise SystemExit("--images must be a multiple of --batch")
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.backends.cudnn.allow_tf32 = False
    ws, bs = lenet_weights(0)
    rng = synth.rng_for(1)
    images = rng.random((a.images, 28, 28), dtype=np.float32)
    paths = {"compressed": Compressed(ws, bs, a.batch), "dense_gemm": DenseGemm(ws, bs, a.batch),
             "dense_cudnn": DenseCudnn(ws, bs, a.batch)}
    errs = cross_check(paths, images[:a.batch])
    dev_images = torch.from_numpy(images).cuda()
    ms = time_paths(paths, dev_images, a.batch, a.reps)
    out = {
        "workload": "LeNet-5 inference, 28x28 synthetic images",
        "images": a.images, "batch": a.batch,
        "nnz": list(SPC_NNZ), "weights": [m * k for m, k in SHAPES],
        "ms": {k: round(v, 4) for k, v in ms.items()},
        "images_per_s": {k: round(a.images / (v / 1e3), 1) for k, v in ms.items()},
        "speedup_vs_dense_gemm": round(ms["dense_gemm"] / ms["compressed"], 3),
        "speedup_vs_dense_cudnn": round(ms["dense_cudnn"] / ms["compressed"], 3),
        "max_rel_diff_vs_compressed": {k: float(f"{v:.3g}") for k, v in errs.items()},
        "paper": PAPER,
    }
    if a.json:
        print(json.dumps(out))
    else:
        for k in ms:
            print(f"{k:<12s} {ms[k]:9.3f} ms for {a.images} images  {out['images_per_s'][k]:14.1f} images/s")
        print(f"speedup of the compressed network: {out['speedup_vs_dense_gemm']}x vs im2col+SGEMM, "
              f"{out['speedup_vs_dense_cudnn']}x vs cuDNN (paper: 2x GTX 1080 Ti, 1.2x Mali-T860)")
    return 0


if __name__ == "__main__":
    sys.exit(main())
