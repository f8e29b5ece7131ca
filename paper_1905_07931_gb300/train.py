"""The CSR-weight training step over a network of sparse layers.

A network is a list of layers, each a dict with ``kind`` in
{"fc", "conv", "pool2", "flatten"} (fc: {"relu"}, conv: {"k", "in_shape",
"relu"}). Weights of fc and conv layers are CSR matrices (Section 3.1);
convolutions are lowered to a matrix product with im2col. One step
(Section 2.3 with a minibatch gradient):

  forward   per layer: [im2col] -> spmm_fwd -> bias (+ ReLU) -> [pool/flatten]
  loss      softmax cross-entropy; dL/dlogits = (softmax - onehot) / B
  backward  per layer, last to first: [ReLU backward] -> weight gradient
            (prox phase: dense G = dY X^T; debias phase: SDDMM at the stored
            entries) -> bias SGD -> spmm_bwd_t (not for the first layer)
            [-> col2im] -> weight update right away, while G is hot in L2:
            prox phase: prox_update_compact into the other CSR buffer
            (Eq. prox, compaction after every update, Section 4.4);
            debias phase: debias_update in place (Section 2.4).

Every buffer is allocated up front, every call is enqueued on one stream and
nothing synchronises, so a step can be captured in a CUDA graph. This module
only sequences calls into the CUDA library.
"""

from __future__ import annotations

import numpy as np
import torch

from . import csrtrain as C


class SparseNet:
    def __init__(self, layers, dense_weights, biases, batch: int, in_shape, *, device="cuda",
                 precision: int = C.CSRT_PREC_TF32, stream=None, grad_per_layer: bool = False,
                 fused: bool = True, optimizer: str = "sgd", beta1: float = 0.9, beta2: float = 0.999,
                 rms_beta: float = 0.9, eps: float = 1e-8, overlap: bool = False):
        """layers: layer dicts; dense_weights/biases: numpy arrays, one per fc/conv
        layer (weights M x K, zero off the initial pattern); in_shape: (K,) for an
        fc-first net or (C, H, W) for a conv-first net. The dense gradients of
        all layers share one buffer unless grad_per_layer is set (then each
        layer's G stays readable after the step).

        optimizer selects the proximal method of the prox phase: "sgd" (the
        proximal gradient step), "rmsprop" (Prox-RMSProp, Algorithm 1, decay
        rms_beta) or "adam" (Prox-ADAM, Algorithm 2, decays beta1 and beta2);
        eps is the safeguard of both. The adaptive methods keep dense M x K
        moment arrays per layer and count their steps on the host (the step
        number is passed by value, so a captured graph replays the step it was
        captured at). The debias phase is plain SGD in every case.

        overlap: in the prox phase, the bias update and the weight update of
        every layer but the first run on a second stream (with its own
        workspace and gradient buffer), concurrently with the transposed
        products that carry dL/dX down the network: the weight update of a
        layer reads its current CSR and writes the other buffer, the
        transposed product only reads the current one. The second stream
        joins the caller's at the end of the step. (The debias phase updates
        the stored values in place and stays on one stream.)"""
        if optimizer not in ("sgd", "rmsprop", "adam"):
            raise ValueError(f"unknown optimizer {optimizer!r}")
        self.optimizer = optimizer
        self.beta1, self.beta2, self.rms_beta, self.eps = beta1, beta2, rms_beta, eps
        self.t = 0
        self.grad_per_layer = grad_per_layer
        # the SGD prox phase applies the update in the gradient GEMM's epilogue
        # (G is not written) unless each layer's G is to stay readable
        self.fused = fused and not grad_per_layer and optimizer == "sgd"
        self.layers = [dict(l) for l in layers]
        self.batch = int(batch)
        self.device = device
        self.precision = precision
        self.stream = stream
        B = self.batch
        dev = dict(device=device, dtype=torch.float32)
        if len(in_shape) == 1:
            self.x_in = torch.zeros(in_shape[0], B, **dev)
        else:
            c, h, w = in_shape
            self.x_in = torch.zeros(c, B * h * w, **dev)
        self.labels = torch.zeros(B, dtype=torch.int32, device=device)
        shape = tuple(in_shape)           # (K,) or (C, H, W) per sample
        cur = self.x_in
        wi = 0
        max_rows = max_cols = max_n = 1
        max_mk = 1
        first_param = True
        self.params = []
        for L in self.layers:
            kind = L["kind"]
            L["x"] = cur
            if kind in ("fc", "conv"):
                W0 = np.ascontiguousarray(dense_weights[wi], dtype=np.float32)
                M, K = W0.shape
                L["needs_dx"] = not first_param
                first_param = False
                L["W"] = [C.CSR(M, K, transposed=L["needs_dx"], device=device),
                          C.CSR(M, K, transposed=L["needs_dx"], device=device)]
                L["cur"] = 0
                L["b"] = torch.tensor(np.asarray(biases[wi], dtype=np.float32), device=device)
                L["W0"] = torch.from_numpy(W0).to(device)
                if kind == "fc":
                    if shape != (K,):
                        raise ValueError(f"fc layer expects {K} inputs, got {shape}")
                    n = B
                    L["xmat"] = cur
                    shape = (M,)
                else:
                    ci, h, w = L["in_shape"]
                    k = L["k"]
                    if shape != (ci, h, w) or K != ci * k * k:
                        raise ValueError(f"conv layer shape mismatch: {shape} vs {(ci, h, w)}")
                    ho, wo = h - k + 1, w - k + 1
                    n = B * ho * wo
                    L["cols"] = torch.zeros(K, n, **dev)
                    L["xmat"] = L["cols"]
                    if L["needs_dx"]:
                        L["dcols"] = torch.zeros(K, n, **dev)
                    shape = (M, ho, wo)
                L["y"] = torch.zeros(M, n, **dev)
                L["dy"] = torch.zeros(M, n, **dev)
                if L["needs_dx"]:
                    L["dx"] = torch.zeros_like(cur)
                L["g"] = torch.zeros(M * K, **dev)
                if optimizer == "adam":
                    L["m"] = torch.zeros(M, K, **dev)
                if optimizer != "sgd":
                    L["v"] = torch.zeros(M, K, **dev)
                if grad_per_layer:
                    L["G"] = torch.zeros(M, K, **dev)
                max_rows, max_cols, max_n = max(max_rows, M), max(max_cols, K), max(max_n, n)
                max_mk = max(max_mk, M * K)
                cur = L["y"]
                self.params.append(L)
                wi += 1
            elif kind == "pool2":
                c, h, w = shape
                L["shape"] = shape
                L["y"] = torch.zeros(c, B * (h // 2) * (w // 2), **dev)
                L["idx"] = torch.zeros(c * B * (h // 2) * (w // 2), dtype=torch.int8, device=device)
                L["dy"] = torch.zeros_like(L["y"])
                L["dx"] = torch.zeros_like(cur)
                shape = (c, h // 2, w // 2)
                cur = L["y"]
            elif kind == "flatten":
                c, h, w = shape
                L["shape"] = shape
                L["y"] = torch.zeros(c * h * w, B, **dev)
                L["dy"] = torch.zeros_like(L["y"])
                L["dx"] = torch.zeros_like(cur)
                shape = (c * h * w,)
                cur = L["y"]
            else:
                raise ValueError(kind)
        self.logits = cur
        self.classes = shape[0]
        self.dlogits = torch.zeros_like(cur)
        self.loss = torch.zeros(B + 1, **dev)
        self.G = torch.zeros(max_mk, **dev)
        self.ws = C.Workspace(max_rows, max_cols, max_n, device=device, stream=stream)
        self.overlap = overlap
        if overlap:
            self.side = torch.cuda.Stream(device=device)
            self.ws_side = C.Workspace(max_rows, max_cols, max_n, device=device, stream=stream)
            self.G_side = torch.zeros(max_mk, **dev)
            n_fc = sum(1 for L in self.layers if L["kind"] in ("fc", "conv"))
            self._events = [torch.cuda.Event() for _ in range(n_fc + 1)]
        for L in self.params:
            C.csr_from_dense(L["W0"], L["W"][0], self.ws, stream)

    # ------------------------------------------------------------------
    def status(self):
        """Device status of the step (synchronises): the flags of every
        workspace the network uses, OR-ed, and the largest required nnz."""
        flags, req = self.ws.status(self.stream)
        if self.overlap:
            f2, r2 = self.ws_side.status(self.stream)
            flags, req = flags | f2, max(req, r2)
        return flags, req

    def weights(self, li: int) -> C.CSR:
        L = self.params[li]
        return L["W"][L["cur"]]

    def set_input(self, x_in: torch.Tensor, labels: torch.Tensor):
        """Point the network at other device buffers for its input batch and
        labels (same shapes and dtypes as ``x_in`` / ``labels``); a step
        captured in a graph afterwards reads them directly."""
        if x_in.shape != self.x_in.shape or x_in.dtype != self.x_in.dtype or x_in.device != self.x_in.device:
            raise ValueError(f"input {tuple(x_in.shape)} {x_in.dtype} does not match {tuple(self.x_in.shape)}")
        if labels.shape != self.labels.shape or labels.dtype != self.labels.dtype:
            raise ValueError("labels do not match")
        if not (x_in.is_contiguous() and labels.is_contiguous()):
            raise ValueError("input buffers must be contiguous")
        old = self.x_in
        for L in self.layers:
            for key in ("x", "xmat"):
                if L.get(key) is old:
                    L[key] = x_in
        self.x_in, self.labels = x_in, labels

    def forward(self):
        s = self.stream
        for L in self.layers:
            kind = L["kind"]
            if kind == "fc":
                W = L["W"][L["cur"]]
                C.spmm_fwd_bias_act(W, L["x"], L["b"], L["relu"], L["y"], self.ws, s)
            elif kind == "conv":
                ci, h, w = L["in_shape"]
                C.im2col(L["x"], ci, self.batch, h, w, L["k"], L["cols"], s)
                W = L["W"][L["cur"]]
                C.spmm_fwd_bias_act(W, L["cols"], L["b"], L["relu"], L["y"], self.ws, s)
            elif kind == "pool2":
                c, h, w = L["shape"]
                C.maxpool2_fwd(L["x"], c, self.batch, h, w, L["y"], L["idx"], s)
            elif kind == "flatten":
                c, h, w = L["shape"]
                C.flatten(L["x"], c, self.batch, h * w, L["y"], s)
        return self.logits

    def step(self, phase: str, eta: float, lam: float):
        """One training step on the data in ``x_in`` / ``labels``. Returns the
        device tensor whose element 0 is the mean loss (not synchronised)."""
        s = self.stream
        if phase == "prox":
            self.t += 1   # step number of the adaptive methods (Algorithms 1 and 2)
        ov = self.overlap and phase == "prox"
        main = (s if s is not None else torch.cuda.current_stream()) if ov else s
        ev_i = 0
        self.forward()
        C.softmax_xent(self.logits, self.labels, self.dlogits, self.loss, s)
        d = self.dlogits
        d_masked = False   # d already carries the ReLU backward of the layer that produced it
        for li in range(len(self.layers) - 1, -1, -1):
            L = self.layers[li]
            kind = L["kind"]
            if kind in ("fc", "conv"):
                W = L["W"][L["cur"]]
                dpre = d
                if L["relu"] and not d_masked:
                    C.relu_bwd(dpre, L["y"], s)
                d_masked = False
                L["dpre"] = dpre   # dL/d(pre-activation) of this layer (a view kept for inspection)
                M, K = W.rows, W.cols
                # this layer's bias and weight update: on the second stream
                # when overlapping (not for the first layer, the last of the step)
                side = ov and L["needs_dx"]
                us, uws = (self.side, self.ws_side) if side else (s, self.ws)
                if side:
                    ev = self._events[ev_i]
                    ev_i += 1
                    ev.record(main)
                    self.side.wait_event(ev)
                if phase == "prox":
                    Gbuf = self.G_side if side else self.G
                    G = L["G"] if self.grad_per_layer else Gbuf[: M * K].view(M, K)
                    if not self.fused:
                        C.weight_grad_dense(dpre, L["xmat"], G, uws, self.precision, us)
                else:
                    C.weight_grad_sddmm(W, dpre, L["xmat"], L["g"], self.ws, s)
                C.bias_grad_sgd(dpre, L["b"], eta, None, us)
                if L["needs_dx"]:
                    below = self.layers[li - 1] if li > 0 else None
                    if kind == "fc" and below is not None and below["kind"] == "fc" and below["relu"]:
                        # ReLU backward of the layer below fused into the transposed product
                        C.spmm_bwd_t_relu(W, dpre, below["y"], L["dx"], self.ws, s)
                        d_masked = True
                    elif kind == "fc":
                        C.spmm_bwd_t(W, dpre, L["dx"], self.ws, s)
                    else:
                        ci, h, w = L["in_shape"]
                        C.spmm_bwd_t(W, dpre, L["dcols"], self.ws, s)
                        C.col2im(L["dcols"], ci, self.batch, h, w, L["k"], L["dx"], s)
                if phase == "prox":
                    Wn = L["W"][1 - L["cur"]]
                    if self.fused:
                        C.weight_grad_prox_update(W, dpre, L["xmat"], eta, lam, Wn, uws, self.precision, G, us)
                    elif self.optimizer == "rmsprop":
                        C.prox_rmsprop_update_compact(W, G, L["v"], eta, lam, self.rms_beta, self.eps, Wn, uws, us)
                    elif self.optimizer == "adam":
                        C.prox_adam_update_compact(W, G, L["m"], L["v"], self.t, eta, lam, self.beta1, self.beta2,
                                                   self.eps, Wn, uws, us)
                    else:
                        C.prox_update_compact(W, G, eta, lam, Wn, uws, us)
                    L["cur"] = 1 - L["cur"]
                else:
                    C.debias_update(W, L["g"], eta, s)
                if not L["needs_dx"]:
                    break
                d = L["dx"]
            elif kind == "pool2":
                c, h, w = L["shape"]
                C.maxpool2_bwd(d, L["idx"], c, self.batch, h, w, L["dx"], s)
                d = L["dx"]
            elif kind == "flatten":
                c, h, w = L["shape"]
                C.unflatten(d, c, self.batch, h * w, L["dx"], s)
                d = L["dx"]
        if ov and ev_i:   # the second stream's work is part of the step
            ev = self._events[ev_i]
            ev.record(self.side)
            main.wait_event(ev)
        return self.loss

    def reset_weights(self):
        """Rebuild every layer's CSR (buffer 0) from its initial dense weights."""
        for L in self.params:
            L["cur"] = 0
            C.csr_from_dense(L["W0"], L["W"][0], self.ws, self.stream)

    def reset_optimizer(self):
        """Zero the adaptive moments and the step counter."""
        self.t = 0
        for L in self.params:
            for key in ("m", "v"):
                if key in L:
                    L[key].zero_()


class BatchPrefetcher:
    """Input pipeline of a SparseNet: batch i+1 is copied from pinned host
    memory into one of two device slots on a copy stream while step i runs.
    Two ways to hand a slot to the network:

    * ``load()``: a device-to-device copy into the network's ``x_in`` /
      ``labels`` on its stream (the network keeps reading ``x_in`` until its
      last weight gradient, so the next batch cannot be copied into ``x_in``
      itself while a step is in flight);
    * ``acquire()`` / ``release(slot)``: the step reads the slot's buffers
      directly (``net.set_input(pf.x[slot], pf.y[slot])``, e.g. one captured
      graph per slot), no copy.

      pf.issue(x0, y0, after=start_event)            # batch 0
      for i in range(steps):
          pf.load()                                   # waits for batch i's copy
          if i + 1 < steps: pf.issue(x[i+1], y[i+1])  # overlaps step i
          net.step(...)
    """

    def __init__(self, net):
        self.net = net
        self.copy_stream = torch.cuda.Stream(device=net.x_in.device)
        self.x = [torch.empty_like(net.x_in) for _ in range(2)]
        self.y = [torch.empty_like(net.labels) for _ in range(2)]
        self.ready = [torch.cuda.Event() for _ in range(2)]
        self.free = [torch.cuda.Event() for _ in range(2)]
        self.issued = 0
        self.loaded = 0

    def _stream(self):
        return self.net.stream or torch.cuda.current_stream()

    def issue(self, x_host: torch.Tensor, y_host: torch.Tensor, after: torch.cuda.Event | None = None):
        """Enqueue the host-to-device copy of the next batch (pinned host
        tensors of the shapes of ``x_in`` and ``labels``); the copy starts
        after ``after`` (an event on the network's stream) if given, and after
        the slot's previous batch has been released."""
        slot = self.issued % 2
        cs = self.copy_stream
        if after is not None:
            cs.wait_event(after)
        cs.wait_event(self.free[slot])
        with torch.cuda.stream(cs):
            self.x[slot].copy_(x_host.view(self.x[slot].shape), non_blocking=True)
            self.y[slot].copy_(y_host, non_blocking=True)
            self.ready[slot].record(cs)
        self.issued += 1

    def acquire(self) -> int:
        """Make the network's stream wait for the oldest issued batch; returns
        its slot (the step then reads ``x[slot]`` / ``y[slot]``)."""
        if self.loaded >= self.issued:
            raise RuntimeError("no batch issued")
        slot = self.loaded % 2
        self._stream().wait_event(self.ready[slot])
        self.loaded += 1
        return slot

    def release(self, slot: int):
        """The work that reads the slot is enqueued: its next copy may follow it."""
        self.free[slot].record(self._stream())

    def load(self):
        """Make the oldest issued batch the network's input (copied into
        ``x_in`` / ``labels`` on its stream)."""
        slot = self.acquire()
        s = self._stream()
        with torch.cuda.stream(s):
            self.net.x_in.copy_(self.x[slot])
            self.net.labels.copy_(self.y[slot])
        self.release(slot)


def mlp_layers(n_layers: int):
    return [{"kind": "fc", "relu": i < n_layers - 1} for i in range(n_layers)]


def lenet_layers():
    return [{"kind": "conv", "k": 5, "in_shape": (1, 28, 28), "relu": False},
            {"kind": "pool2"},
            {"kind": "conv", "k": 5, "in_shape": (20, 12, 12), "relu": False},
            {"kind": "pool2"},
            {"kind": "flatten"},
            {"kind": "fc", "relu": True},
            {"kind": "fc", "relu": False}]


class SingleLayer:
    """The single-layer step (one CSR layer, upstream gradient given):
    forward SpMM, backward SpMM^T, dense weight gradient, prox + compaction."""

    def __init__(self, w_dense: np.ndarray, n: int, device="cuda", precision: int = C.CSRT_PREC_TF32,
                 stream=None):
        M, K = w_dense.shape
        self.stream = stream
        self.precision = precision
        self.W = [C.CSR(M, K, device=device), C.CSR(M, K, device=device)]
        self.cur = 0
        self.W0 = torch.from_numpy(np.ascontiguousarray(w_dense, dtype=np.float32)).to(device)
        self.x = torch.zeros(K, n, device=device)
        self.dy = torch.zeros(M, n, device=device)
        self.y = torch.zeros(M, n, device=device)
        self.dx = torch.zeros(K, n, device=device)
        self.G = torch.zeros(M, K, device=device)
        self.ws = C.Workspace(M, K, n, device=device, stream=stream)
        C.csr_from_dense(self.W0, self.W[0], self.ws, stream)

    def step(self, eta: float, lam: float):
        s = self.stream
        W = self.W[self.cur]
        C.spmm_fwd(W, self.x, self.y, self.ws, s)
        C.spmm_bwd_t(W, self.dy, self.dx, self.ws, s)
        C.weight_grad_dense(self.dy, self.x, self.G, self.ws, self.precision, s)
        C.prox_update_compact(W, self.G, eta, lam, self.W[1 - self.cur], self.ws, s)
        self.cur = 1 - self.cur
