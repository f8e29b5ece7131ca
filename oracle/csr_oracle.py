"""Plain CPU restatement of the CSR-weight training step (test infrastructure).

Every function here follows a definition stated in the paper (Lee & Lee,
arXiv 1905.07931) or, for the network glue the paper inherits from Caffe
without describing it, the textbook definition of that layer. Nothing here is
blocked, fused or reordered beyond the definition; library primitives
(``numpy`` dot products, ``nonzero``, ``lexsort``) serve as single steps.

Layout used throughout (the paper's Caffe orientation transposed, Section 3.2):
  * W is M x K (M outputs, K inputs) held in CSR (Section 3.1): ``row_ptr``
    [M+1] int32, ``col_idx`` [nnz] int32 ascending within a row, ``val`` [nnz].
  * Activations are feature-major: X is K x N, Y is M x N, the sample index
    (batch, or batch x height x width for a convolution) contiguous.
    Section 3.2 writes the forward pass as X_T = X_B W' with samples in rows;
    with samples in columns the same product is Y = W X.

Sums are accumulated in float64 and returned as float64; callers round to
float32 where they compare. The proximal step and the debias update follow
explicit float32 rounding rules (see their docstrings) so their outputs are
bit-exact.

Readings of the paper taken here (each is also listed in the design notes):
  * The threshold is applied as thr = fl32(eta * lambda) with eta, lambda
    float32 (Section 2.2 with Psi = eta*lambda*||.||_1, Eq. prox).
  * |z| == thr is dropped (both the closed form of Section 2.2 and the min/max
    kernel form of Section 3.3 give exactly zero there); NaN z is dropped.
  * The prox acts on the dense w - eta*G (Section 3.3: the kernel's matrix A
    holds w - eta*G), so zero weights may re-enter.
  * Debiasing (Section 2.4 and 4.3: zero weights are fixed and not updated) is
    plain SGD on the stored entries; the pattern never changes, a stored value
    that reaches 0.0 stays stored.
  * Biases are dense, unregularised, plain SGD.
  * The 1/|B| of the minibatch gradient (Section 2.2) lives in the loss
    gradient: softmax cross-entropy returns (softmax - onehot) / B.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "CSR", "csr_from_dense", "csr_to_dense", "csr_abs", "csr_transpose",
    "spmm_fwd", "spmm_bwd_t", "weight_grad_dense", "weight_grad_sddmm",
    "soft_threshold", "prox_update_compact", "debias_update",
    "rmsprop_direction", "adam_direction", "prox_rmsprop_update_compact", "prox_adam_update_compact",
    "dense_times_compressed_t", "dense_times_compressed",
    "compression_rate",
    "im2col", "col2im", "maxpool2_fwd", "maxpool2_bwd", "relu",
    "softmax_xent", "flatten_cnhw", "unflatten_cnhw",
    "Net", "net_forward", "net_backward", "net_step", "net_loss_dense",
]

F32 = np.float32
F64 = np.float64


# ---------------------------------------------------------------------------
# CSR storage -- Section 3.1 and the worked example of Figure "spformats" (iii)
# ---------------------------------------------------------------------------

@dataclass
class CSR:
    """A compressed sparse row matrix (Section 3.1).

    ``row_ptr[i]`` is the index in ``col_idx``/``val`` where row i begins,
    ``row_ptr[M]`` = nnz. Columns are ascending and unique within a row.
    ``val`` keeps the dtype it was built with (float32 for the product path,
    float64 is allowed for finite-difference checks).
    """

    rows: int
    cols: int
    row_ptr: np.ndarray
    col_idx: np.ndarray
    val: np.ndarray

    @property
    def nnz(self) -> int:
        return int(self.row_ptr[-1])

    def row_of_each_entry(self) -> np.ndarray:
        """COO row array (Figure "spformats" (iv)) derived from row_ptr."""
        lengths = np.diff(self.row_ptr.astype(np.int64))
        return np.repeat(np.arange(self.rows, dtype=np.int64), lengths)


def csr_from_dense(dense: np.ndarray) -> CSR:
    """Keep every entry with value != 0 in row-major order (Section 3.1).

    Rows are scanned top to bottom, columns left to right. ``v != 0`` drops
    +0.0 and -0.0 and keeps NaN and +-Inf. Pinned by the worked example of
    Figure "spformats" (iii) and by brute-force densify/round-trip tests.
    """
    dense = np.asarray(dense)
    if dense.ndim != 2:
        raise ValueError("dense must be 2-D")
    m, k = dense.shape
    keep = dense != 0
    counts = keep.sum(axis=1)
    row_ptr = np.zeros(m + 1, dtype=np.int64)
    row_ptr[1:] = np.cumsum(counts)
    rows, cols = np.nonzero(keep)          # row-major order by definition
    return CSR(m, k, row_ptr.astype(np.int32), cols.astype(np.int32),
               dense[rows, cols].copy())


def csr_to_dense(w: CSR, dtype=None) -> np.ndarray:
    """Dense M x K matrix with the stored values and +0 off the pattern."""
    dtype = w.val.dtype if dtype is None else dtype
    out = np.zeros((w.rows, w.cols), dtype=dtype)
    out[w.row_of_each_entry(), w.col_idx.astype(np.int64)] = w.val
    return out


def csr_abs(w: CSR) -> CSR:
    """Same pattern, |val| (used for the summation error bound sum |terms|)."""
    return CSR(w.rows, w.cols, w.row_ptr, w.col_idx, np.abs(w.val))


def csr_transpose(w: CSR):
    """The transposed pattern: CSR of W^T, i.e. W stored column by column.

    Section 3.2.2 notes that the backward product needs column-wise access
    and that this takes an extra array holding the nonzeros column-wise. That
    array is defined here: entries sorted by (column, row). Returns
    ``(t_row_ptr[K+1], t_col_idx[nnz] (row of each entry), t_val[nnz],
    t_pos[nnz])`` where ``t_pos[k]`` is the transposed position of CSR entry k.
    Pinned by the hand-transposed worked example and by
    ``csr_from_dense(dense.T)``.
    """
    rows = w.row_of_each_entry()
    cols = w.col_idx.astype(np.int64)
    order = np.lexsort((rows, cols))        # primary key column, then row
    t_row_ptr = np.zeros(w.cols + 1, dtype=np.int64)
    t_row_ptr[1:] = np.cumsum(np.bincount(cols, minlength=w.cols))
    t_pos = np.empty(w.nnz, dtype=np.int64)
    t_pos[order] = np.arange(w.nnz)
    return (t_row_ptr.astype(np.int32), rows[order].astype(np.int32),
            w.val[order].copy(), t_pos.astype(np.int32))


# ---------------------------------------------------------------------------
# Sparse x dense products -- Section 3.2 (forward D x C', backward D x C)
# ---------------------------------------------------------------------------

def spmm_fwd(w: CSR, x: np.ndarray) -> np.ndarray:
    """Y = W X, Y[i, n] = sum over stored k of row i of val[k] * X[col[k], n].

    The forward product of Section 3.2 (X_T = X_B W' with samples in rows).
    Accumulated in float64 in CSR order. Pinned by dense brute force, by the
    worked example (A times a vector of ones) and by the Caffe-orientation
    restatement ``dense_times_compressed_t``.
    """
    x = np.asarray(x, dtype=F64)
    if x.shape[0] != w.cols:
        raise ValueError("X must have K rows")
    y = np.zeros((w.rows, x.shape[1]), dtype=F64)
    rp = w.row_ptr
    for i in range(w.rows):
        s, e = int(rp[i]), int(rp[i + 1])
        if e > s:
            y[i] = w.val[s:e].astype(F64) @ x[w.col_idx[s:e]]
    return y


def spmm_bwd_t(w: CSR, dy: np.ndarray) -> np.ndarray:
    """dX = W^T dY, dX[j, n] = sum_i W[i, j] dY[i, n].

    The backward product of Section 3.2 (dL/dX_B = dL/dX_T W with samples in
    rows). Each stored entry (i, j) adds val * dY[i, :] to dX[j, :].
    Pinned by dense brute force, by the worked example (A^T times ones) and by
    ``dense_times_compressed``.
    """
    dy = np.asarray(dy, dtype=F64)
    if dy.shape[0] != w.rows:
        raise ValueError("dY must have M rows")
    dx = np.zeros((w.cols, dy.shape[1]), dtype=F64)
    rp = w.row_ptr
    for i in range(w.rows):
        s, e = int(rp[i]), int(rp[i + 1])
        if e > s:
            cols = w.col_idx[s:e]           # unique within a row
            dx[cols] += np.outer(w.val[s:e].astype(F64), dy[i])
    return dx


def dense_times_compressed_t(xb: np.ndarray, w: CSR) -> np.ndarray:
    """Section 3.2.1 in the paper's own orientation: result = X_B W'.

    ``xb`` holds one sample per row (N x K). result[row, col] is the inner
    product of sample ``row`` with row ``col`` of W, walked through that row's
    stored entries. Written independently of ``spmm_fwd`` as a cross-check of
    the orientation (double accumulators, as in the paper's kernel).
    """
    xb = np.asarray(xb, dtype=F64)
    n = xb.shape[0]
    out = np.zeros((n, w.rows), dtype=F64)
    for r in range(n):
        for c in range(w.rows):
            acc = 0.0
            for k in range(int(w.row_ptr[c]), int(w.row_ptr[c + 1])):
                acc += xb[r, int(w.col_idx[k])] * float(w.val[k])
            out[r, c] = acc
    return out


def dense_times_compressed(dxt: np.ndarray, w: CSR) -> np.ndarray:
    """Section 3.2.2 in the paper's own orientation: result = dX_T W.

    ``dxt`` holds one sample per row (N x M). result[row, col] sums, over the
    rows i of W that store column ``col``, dX_T[row, i] * W[i, col]. Restated
    from the definition (the paper's listing is a scan over all nonzeros with
    a running row index); it does not reuse ``spmm_bwd_t``.
    """
    dxt = np.asarray(dxt, dtype=F64)
    n = dxt.shape[0]
    out = np.zeros((n, w.cols), dtype=F64)
    rows = w.row_of_each_entry()
    for r in range(n):
        for k in range(w.nnz):
            out[r, int(w.col_idx[k])] += dxt[r, int(rows[k])] * float(w.val[k])
    return out


# ---------------------------------------------------------------------------
# Weight gradients
# ---------------------------------------------------------------------------

def weight_grad_dense(dy: np.ndarray, x: np.ndarray) -> np.ndarray:
    """G = dY X^T, G[i, j] = sum_n dY[i, n] X[j, n] (all M x K entries).

    The gradient of the loss with respect to every weight, zero or not; the
    prox step acts on the dense w - eta*G (Section 3.3). No 1/N factor: the
    loss gradient already carries it. Pinned by finite differences of the
    network loss and by a triple loop on tiny shapes.
    """
    return np.asarray(dy, dtype=F64) @ np.asarray(x, dtype=F64).T


def weight_grad_sddmm(w: CSR, dy: np.ndarray, x: np.ndarray) -> np.ndarray:
    """g[k] = sum_n dY[i_k, n] X[j_k, n] at the stored entries only.

    The debias gradient (Section 2.4: zero weights are excluded from
    training). Pinned by equality with ``weight_grad_dense`` read at the
    pattern and by finite differences at stored entries.
    """
    dy = np.asarray(dy, dtype=F64)
    x = np.asarray(x, dtype=F64)
    g = np.zeros(w.nnz, dtype=F64)
    rp = w.row_ptr
    for i in range(w.rows):
        s, e = int(rp[i]), int(rp[i + 1])
        if e > s:
            g[s:e] = x[w.col_idx[s:e]] @ dy[i]
    return g


# ---------------------------------------------------------------------------
# Proximal step -- Section 2.2 (closed form), Eq. prox (Section 2.3),
# Section 3.3 (applied to the dense w - eta*G), "compression every update"
# (Section 4.4)
# ---------------------------------------------------------------------------

def soft_threshold(z: np.ndarray, thr) -> np.ndarray:
    """sgn(z) * max(|z| - thr, 0), the closed form of Section 2.2.

    Evaluated in float32: for |z| > thr the result is z - thr (z > 0) or
    z + thr (z < 0), each rounded once; otherwise 0.
    """
    z = np.asarray(z, dtype=F32)
    thr = F32(thr)
    mag = np.abs(z) - thr
    out = np.where(mag > 0, np.where(z > 0, z - thr, z + thr), F32(0))
    return out.astype(F32)


def prox_update_compact(w: CSR, g: np.ndarray, eta: float, lam: float) -> CSR:
    """One proximal SGD update followed by CSR re-compaction.

    Eq. prox: w <- prox_{eta*Psi}(w - eta*g) with Psi = lambda*||.||_1, whose
    prox is the soft threshold at eta*lambda (Section 2.2). The update acts on
    all M x K entries (the matrix w - eta*G of Section 3.3; off-pattern w is
    +0), and the result is compacted back to CSR after every update
    (Section 4.4).

    Float32 rules (fixed so that the kept pattern is bit-exact):
      thr = fl32(eta * lambda); t = fl32(eta * G[i,j]); z = fl32(w - t)
      keep iff |z| > thr; kept value = soft_threshold(z, thr).
    Pinned by hand cases with exactly representable values, by agreement with
    the min/max form of Section 3.3, and by the identity/empty/nesting
    properties.
    """
    g = np.asarray(g, dtype=F32)
    if g.shape != (w.rows, w.cols):
        raise ValueError("G must be M x K")
    eta32, lam32 = F32(eta), F32(lam)
    thr = eta32 * lam32
    wd = csr_to_dense(w, dtype=F32)
    t = eta32 * g
    z = wd - t
    keep = np.abs(z) > thr
    out = soft_threshold(z, thr)
    # keep and out != 0 agree: |z| > thr implies |z| - thr > 0 in float32
    # (Sterbenz), so the kept value is never zero.
    dense_new = np.where(keep, out, F32(0)).astype(F32)
    return csr_from_dense(dense_new)


def rmsprop_direction(g: np.ndarray, v: np.ndarray, beta: float, eps: float):
    """The moment update and search direction of one Prox-RMSProp step
    (Algorithm 1), on every M x K entry.

    Algorithm 1 keeps v, the running average of g*g (elementwise), and moves
    along g / (sqrt(v) + eps). Float32 rules, every operation rounded once,
    in this order (c = fl32(1 - beta)):
      v' = fl(fl(beta * v) + fl(c * fl(g * g)))
      d  = fl(g / fl(fl(sqrt(v')) + eps))
    Returns (v', d). Pinned by exact hand cases, by the beta = 0 reduction
    shared with Adam, and by a five-step trajectory against the textbook
    float64 method.
    """
    g = np.asarray(g, dtype=F32)
    v = np.asarray(v, dtype=F32)
    beta32, eps32 = F32(beta), F32(eps)
    c = F32(1) - beta32
    v_new = (beta32 * v + c * (g * g)).astype(F32)
    d = (g / (np.sqrt(v_new) + eps32)).astype(F32)
    return v_new, d


def adam_direction(g: np.ndarray, m: np.ndarray, v: np.ndarray, t: int, beta1: float, beta2: float,
                   eps: float):
    """The moment updates and search direction of step t >= 1 of Prox-ADAM
    (Algorithm 2), on every M x K entry.

    Algorithm 2 keeps the first moment m and the second moment v of g, divides
    each by its bias correction 1 - beta^t, and moves along
    m_hat / (sqrt(v_hat) + eps). Float32 rules, every operation rounded once,
    in this order (c_i = fl32(1 - beta_i); the corrections bc_i =
    fl32(1 - beta_i^t) with the power taken in float64):
      m' = fl(fl(beta1 * m) + fl(c1 * g))
      v' = fl(fl(beta2 * v) + fl(c2 * fl(g * g)))
      m_hat = fl(m' / bc1), v_hat = fl(v' / bc2)
      d = fl(m_hat / fl(fl(sqrt(v_hat)) + eps))
    Returns (m', v', d). Pinned like rmsprop_direction.
    """
    if int(t) < 1:
        raise ValueError("the step counter t starts at 1")
    g = np.asarray(g, dtype=F32)
    m = np.asarray(m, dtype=F32)
    v = np.asarray(v, dtype=F32)
    b1, b2, eps32 = F32(beta1), F32(beta2), F32(eps)
    c1, c2 = F32(1) - b1, F32(1) - b2
    bc1 = F32(1.0 - float(b1) ** int(t))
    bc2 = F32(1.0 - float(b2) ** int(t))
    m_new = (b1 * m + c1 * g).astype(F32)
    v_new = (b2 * v + c2 * (g * g)).astype(F32)
    m_hat = (m_new / bc1).astype(F32)
    v_hat = (v_new / bc2).astype(F32)
    d = (m_hat / (np.sqrt(v_hat) + eps32)).astype(F32)
    return m_new, v_new, d


def prox_rmsprop_update_compact(w: CSR, g: np.ndarray, v: np.ndarray, eta: float, lam: float, beta: float,
                                eps: float):
    """One Prox-RMSProp step (Algorithm 1) followed by CSR re-compaction:
    w <- prox_{eta*lambda*||.||_1}(w - eta * d) with d from rmsprop_direction,
    i.e. prox_update_compact applied to d (the threshold stays eta*lambda, not
    scaled by the adaptive denominator). Returns (w', v')."""
    v_new, d = rmsprop_direction(g, v, beta, eps)
    return prox_update_compact(w, d, eta, lam), v_new


def prox_adam_update_compact(w: CSR, g: np.ndarray, m: np.ndarray, v: np.ndarray, t: int, eta: float,
                             lam: float, beta1: float, beta2: float, eps: float):
    """One Prox-ADAM step (Algorithm 2) followed by CSR re-compaction:
    w <- prox_{eta*lambda*||.||_1}(w - eta * d) with d from adam_direction.
    Returns (w', m', v')."""
    m_new, v_new, d = adam_direction(g, m, v, t, beta1, beta2, eps)
    return prox_update_compact(w, d, eta, lam), m_new, v_new


def debias_update(w: CSR, g: np.ndarray, eta: float) -> CSR:
    """Debias (retraining) step on stored entries: val <- fl32(val - fl32(eta*g)).

    Section 2.4 / Section 4.3: no regulariser, the zero weights stay fixed and
    are not updated, so ``row_ptr`` and ``col_idx`` are returned unchanged
    (a value that becomes 0.0 stays stored).
    """
    eta32 = F32(eta)
    g = np.asarray(g, dtype=F32)
    new_val = (w.val.astype(F32) - eta32 * g).astype(F32)
    return CSR(w.rows, w.cols, w.row_ptr.copy(), w.col_idx.copy(), new_val)


def compression_rate(w: CSR) -> float:
    """(number of zero entries) / (number of parameters) (Section 4.1)."""
    total = w.rows * w.cols
    return 1.0 - w.nnz / total if total else 0.0


# ---------------------------------------------------------------------------
# Network glue the paper inherits from Caffe (not described in the paper):
# convolution lowered to a matrix product, max pooling, ReLU, bias, softmax
# cross-entropy, flatten. Activations of convolutional layers are held as
# arrays (C, B, H, W) = a C x (B*H*W) matrix in feature-major order.
# ---------------------------------------------------------------------------

def im2col(x: np.ndarray, k: int) -> np.ndarray:
    """Unfold (C, B, H, W) into (C*k*k) x (B*Ho*Wo), stride 1, no padding.

    Row c*k*k + ky*k + kx, column b*Ho*Wo + oy*Wo + ox holds
    x[c, b, oy+ky, ox+kx]. Pinned by a direct-convolution loop.
    """
    c, b, h, w = x.shape
    ho, wo = h - k + 1, w - k + 1
    cols = np.empty((c, k, k, b, ho, wo), dtype=x.dtype)
    for ky in range(k):
        for kx in range(k):
            cols[:, ky, kx] = x[:, :, ky:ky + ho, kx:kx + wo]
    return cols.reshape(c * k * k, b * ho * wo)


def col2im(dcols: np.ndarray, c: int, b: int, h: int, w: int, k: int) -> np.ndarray:
    """Adjoint of ``im2col``: sum every column entry back onto its pixel."""
    ho, wo = h - k + 1, w - k + 1
    d = np.asarray(dcols, dtype=F64).reshape(c, k, k, b, ho, wo)
    dx = np.zeros((c, b, h, w), dtype=F64)
    for ky in range(k):
        for kx in range(k):
            dx[:, :, ky:ky + ho, kx:kx + wo] += d[:, ky, kx]
    return dx


def maxpool2_fwd(x: np.ndarray):
    """2x2 max pooling, stride 2, on (C, B, H, W) with H and W even.

    Returns (y, idx) with idx in {0,1,2,3} = dy*2 + dx of the first maximum in
    the scan order (0,0), (0,1), (1,0), (1,1).
    """
    c, b, h, w = x.shape
    win = x.reshape(c, b, h // 2, 2, w // 2, 2).transpose(0, 1, 2, 4, 3, 5)
    win = win.reshape(c, b, h // 2, w // 2, 4)
    idx = np.argmax(win, axis=-1)            # first occurrence of the maximum
    y = np.take_along_axis(win, idx[..., None], axis=-1)[..., 0]
    return y, idx.astype(np.int8)


def maxpool2_bwd(dy: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Route each pooled gradient to the window position that won."""
    c, b, ho, wo = dy.shape
    dwin = np.zeros((c, b, ho, wo, 4), dtype=F64)
    np.put_along_axis(dwin, idx.astype(np.int64)[..., None],
                      np.asarray(dy, dtype=F64)[..., None], axis=-1)
    dwin = dwin.reshape(c, b, ho, wo, 2, 2).transpose(0, 1, 2, 4, 3, 5)
    return dwin.reshape(c, b, ho * 2, wo * 2)


def relu(x: np.ndarray) -> np.ndarray:
    return np.maximum(x, 0)


def softmax_xent(z: np.ndarray, labels: np.ndarray):
    """Mean softmax cross-entropy over the N columns of z (C x N).

    Returns (loss, dz) with dz = (softmax(z) - onehot(labels)) / N, the
    minibatch mean of Section 2.2.
    """
    z = np.asarray(z, dtype=F64)
    c, n = z.shape
    zmax = z.max(axis=0, keepdims=True)
    e = np.exp(z - zmax)
    p = e / e.sum(axis=0, keepdims=True)
    lab = np.asarray(labels, dtype=np.int64)
    logp = (z - zmax) - np.log(e.sum(axis=0, keepdims=True))
    loss = -logp[lab, np.arange(n)].mean() if n else 0.0
    dz = p.copy()
    dz[lab, np.arange(n)] -= 1.0
    return float(loss), dz / max(n, 1)


def flatten_cnhw(x: np.ndarray) -> np.ndarray:
    """(C, B, h, w) -> (C*h*w) x B, feature index c*h*w + y*w + x (Caffe order)."""
    c, b, h, w = x.shape
    return x.transpose(0, 2, 3, 1).reshape(c * h * w, b)


def unflatten_cnhw(xf: np.ndarray, c: int, b: int, h: int, w: int) -> np.ndarray:
    """Inverse permutation of ``flatten_cnhw``."""
    return np.asarray(xf).reshape(c, h, w, b).transpose(0, 3, 1, 2)


# ---------------------------------------------------------------------------
# Networks: a list of layers, one training step (Section 2.3 update with the
# minibatch gradient, then either the prox update (sparse coding phase) or the
# debias update (retraining phase, Section 2.4)).
# ---------------------------------------------------------------------------

@dataclass
class Net:
    """Layer list. Each layer is a dict with ``kind`` in
    {"fc", "conv", "pool2", "flatten"}:
      fc:      {"relu": bool}
      conv:    {"k": int, "in_shape": (C, H, W), "relu": bool}
      pool2:   {}
      flatten: {}
    Parameters live in ``params``: per fc/conv layer {"W": CSR, "b": array}.
    """

    layers: list
    params: list = field(default_factory=list)


def net_forward(net: Net, x0: np.ndarray, batch: int):
    """Forward pass. ``x0`` is the input as a feature-major matrix
    (features x batch) for an fc-first net, or (C, B, H, W) for a conv-first
    net. Returns (logits, cache)."""
    cache = []
    x = np.asarray(x0, dtype=F64)
    for layer, p in zip(net.layers, net.params):
        kind = layer["kind"]
        if kind == "fc":
            pre = spmm_fwd(p["W"], x) + np.asarray(p["b"], dtype=F64)[:, None]
            y = relu(pre) if layer["relu"] else pre
            cache.append({"x": x, "pre": pre})
            x = y
        elif kind == "conv":
            c, h, w = layer["in_shape"]
            k = layer["k"]
            xin = x.reshape(c, batch, h, w)
            cols = im2col(xin, k)
            pre = spmm_fwd(p["W"], cols) + np.asarray(p["b"], dtype=F64)[:, None]
            y = relu(pre) if layer["relu"] else pre
            cout = p["W"].rows
            cache.append({"x": cols, "pre": pre})
            x = y.reshape(cout, batch, h - k + 1, w - k + 1)
        elif kind == "pool2":
            y, idx = maxpool2_fwd(x)
            cache.append({"idx": idx, "shape": x.shape})
            x = y
        elif kind == "flatten":
            cache.append({"shape": x.shape})
            x = flatten_cnhw(x)
        else:
            raise ValueError(kind)
    return x, cache


def net_backward(net: Net, cache, dz: np.ndarray, phase: str):
    """Backward pass from dL/dlogits. Returns per-layer dicts with
    ``G`` (dense weight gradient, prox phase) or ``g`` (gradient at stored
    entries, debias phase), ``gb`` (bias gradient), ``delta`` (dL/dpre) and
    ``x`` (the layer's matrix input)."""
    grads = [None] * len(net.layers)
    d = np.asarray(dz, dtype=F64)
    first_param = next(i for i, l in enumerate(net.layers) if l["kind"] in ("fc", "conv"))
    for li in range(len(net.layers) - 1, -1, -1):
        layer, p, c = net.layers[li], net.params[li], cache[li]
        kind = layer["kind"]
        if kind in ("fc", "conv"):
            pre = c["pre"]
            if kind == "conv":
                d = d.reshape(p["W"].rows, -1)
            delta = d * (pre > 0) if layer["relu"] else d
            gr = {"delta": delta, "x": c["x"], "gb": delta.sum(axis=1)}
            if phase == "prox":
                gr["G"] = weight_grad_dense(delta, c["x"])
            else:
                gr["g"] = weight_grad_sddmm(p["W"], delta, c["x"])
            grads[li] = gr
            if li > first_param:
                dx = spmm_bwd_t(p["W"], delta)
                if kind == "conv":
                    cin, h, w = layer["in_shape"]
                    batch = c["x"].shape[1] // ((h - layer["k"] + 1) * (w - layer["k"] + 1))
                    dx = col2im(dx, cin, batch, h, w, layer["k"])
                d = dx
            else:
                d = None
        elif kind == "pool2":
            cs, b, h, w = c["shape"]
            d = maxpool2_bwd(d.reshape(cs, b, h // 2, w // 2), c["idx"])
        elif kind == "flatten":
            cs, b, h, w = c["shape"]
            d = unflatten_cnhw(d, cs, b, h, w)
        if d is None:
            break
    return grads


def net_step(net: Net, x0, labels, eta: float, lam: float, phase: str):
    """One training step (minibatch gradient then update) in place on ``net``.

    phase "prox": W <- prox_update_compact(W, G, eta, lambda) (Eq. prox).
    phase "debias": W.val <- W.val - eta*g at stored entries (Section 2.4).
    Biases: b <- fl32(b - fl32(eta*gb)) in both phases.
    Returns (loss, grads).
    """
    batch = len(labels)
    logits, cache = net_forward(net, x0, batch)
    loss, dz = softmax_xent(logits, labels)
    grads = net_backward(net, cache, dz, phase)
    eta32 = F32(eta)
    for li, layer in enumerate(net.layers):
        if layer["kind"] not in ("fc", "conv"):
            continue
        p, gr = net.params[li], grads[li]
        if phase == "prox":
            p["W"] = prox_update_compact(p["W"], gr["G"].astype(F32), eta, lam)
        else:
            p["W"] = debias_update(p["W"], gr["g"].astype(F32), eta)
        p["b"] = (np.asarray(p["b"], dtype=F32) - eta32 * gr["gb"].astype(F32)).astype(F32)
    return loss, grads


def net_loss_dense(net: Net, dense_ws, biases, x0, labels) -> float:
    """Loss of the net with the given dense weight matrices (float64), for
    finite-difference checks: each dense matrix is re-compressed with
    ``csr_from_dense`` so perturbing a zero entry adds it to the pattern."""
    params = []
    wi = 0
    for layer in net.layers:
        if layer["kind"] in ("fc", "conv"):
            params.append({"W": csr_from_dense(np.asarray(dense_ws[wi], dtype=F64)),
                           "b": np.asarray(biases[wi], dtype=F64)})
            wi += 1
        else:
            params.append(None)
    logits, _ = net_forward(Net(net.layers, params), x0, len(labels))
    loss, _ = softmax_xent(logits, labels)
    return loss
