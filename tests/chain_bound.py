"""Element-wise error bounds for a whole forward / backward chain.

A GPU step computes every layer in float32 from the float32 results of the
layer before; the oracle computes the same chain in float64. Their difference
at each element is bounded by carrying, layer by layer, a bound F (forward)
or E (backward) on the error of every element:

  product  y = W x + b:   F_y = |W| F_x + gamma_{len+2} (|W| (|x| + F_x) + |b|)
           (any summation order; len = stored entries of the row)
  ReLU, max pooling, im2col, flatten: 1-Lipschitz or copies, F carried over
           (max pooling: the largest F of the window)
  softmax: with eps = max_j F_z[j] of a column, p_gpu / p lies within
           exp(+-2 eps), so |dp| <= p (exp(2 eps) - 1), plus float32 rounding
  backward product dX = W^T dY: E_x = |W|^T E + gamma_{clen+1} |W|^T (|dY| + E)
  ReLU backward: where |pre| <= F_pre the two masks may differ, and either
           0 or the passed gradient is right: E there is |d| + E
  col2im:  E_x = col2im(E) + gamma_{k*k} col2im(|d| + E)

Each step is a true upper bound (not first order): the products use the
worst-case summation bound, which holds for every order of summation. The
oracle functions supply every product; this module only combines them.
"""

from __future__ import annotations

import numpy as np

import oracle as O
from tests.parity import U32, gamma


def _product_bound(W, x, Fx, b):
    absW = O.csr_abs(W)
    lens = np.diff(W.row_ptr.astype(np.int64))[:, None]
    S = O.spmm_fwd(absW, np.abs(x) + Fx) + np.abs(np.asarray(b, dtype=np.float64))[:, None]
    return O.spmm_fwd(absW, Fx) + gamma(lens + 2) * S


def _window_max(F):
    c, b, h, w = F.shape
    return F.reshape(c, b, h // 2, 2, w // 2, 2).max(axis=(3, 5))


def forward_bounds(net: "O.Net", x0, batch: int, pool_idx=None):
    """Oracle forward of ``net`` with a bound on each layer's GPU output.

    Returns (logits, F_logits, per_layer) where per_layer[li] holds, for fc
    and conv layers, ``pre`` (float64 pre-activation) and ``F_pre``; for
    pool layers ``idx`` (the winners used for routing: ``pool_idx[li]`` if
    given, e.g. the GPU's where it picked another of tied maxima) and
    ``shape``; for flatten ``shape``."""
    x = np.asarray(x0, dtype=np.float64)
    F = np.zeros_like(x)
    per = []
    for li, (layer, p) in enumerate(zip(net.layers, net.params)):
        kind = layer["kind"]
        if kind in ("fc", "conv"):
            if kind == "conv":
                c, h, w = layer["in_shape"]
                k = layer["k"]
                x = O.im2col(x.reshape(c, batch, h, w), k)
                F = O.im2col(F.reshape(c, batch, h, w), k)
            pre = O.spmm_fwd(p["W"], x) + np.asarray(p["b"], dtype=np.float64)[:, None]
            F_pre = _product_bound(p["W"], x, F, p["b"])
            per.append({"pre": pre, "F_pre": F_pre, "x": x, "F_x": F})
            y = O.relu(pre) if layer["relu"] else pre
            x, F = y, F_pre
            if kind == "conv":
                c, h, w = layer["in_shape"]
                k = layer["k"]
                shape = (p["W"].rows, batch, h - k + 1, w - k + 1)
                x, F = x.reshape(shape), F.reshape(shape)
        elif kind == "pool2":
            y, idx = O.maxpool2_fwd(x)
            if pool_idx is not None and pool_idx.get(li) is not None:
                idx = pool_idx[li]
            per.append({"idx": idx, "shape": x.shape})
            x, F = y, _window_max(F)
        elif kind == "flatten":
            per.append({"shape": x.shape})
            x, F = O.flatten_cnhw(x), O.flatten_cnhw(F)
        else:
            raise ValueError(kind)
    return x, F, per


def softmax_bound(logits, F_logits, labels):
    """Oracle dL/dlogits and a bound on the GPU's."""
    _, dz = O.softmax_xent(logits, labels)
    classes, n = logits.shape
    z = logits - logits.max(axis=0, keepdims=True)
    p = np.exp(z) / np.exp(z).sum(axis=0, keepdims=True)
    eps = F_logits.max(axis=0, keepdims=True)
    dp = p * np.expm1(2.0 * eps) + 8.0 * (classes + 4) * U32 * p + 4.0 * U32
    return dz, dp / max(n, 1) + U32 * np.abs(dz)


def backward_bounds(net: "O.Net", per, dz, E_dz, batch: int):
    """Oracle dL/dpre of every fc / conv layer with a bound on the GPU's.

    Returns {layer index: (delta, E_delta)}."""
    out = {}
    d, E = np.asarray(dz, dtype=np.float64), np.asarray(E_dz, dtype=np.float64)
    first = next(i for i, l in enumerate(net.layers) if l["kind"] in ("fc", "conv"))
    for li in range(len(net.layers) - 1, -1, -1):
        layer, p, c = net.layers[li], net.params[li], per[li]
        kind = layer["kind"]
        if kind in ("fc", "conv"):
            W = p["W"]
            d, E = d.reshape(W.rows, -1), E.reshape(W.rows, -1)
            if layer["relu"]:
                on = c["pre"] > 0
                ambiguous = np.abs(c["pre"]) <= c["F_pre"]
                d, E = d * on, np.where(ambiguous, np.abs(d) + E, E * on)
            out[li] = (d, E)
            if li == first:
                break
            absW = O.csr_abs(W)
            clens = np.bincount(W.col_idx, minlength=W.cols)[:, None]
            dx = O.spmm_bwd_t(W, d)
            Ex = O.spmm_bwd_t(absW, E) + gamma(clens + 1) * O.spmm_bwd_t(absW, np.abs(d) + E)
            if kind == "conv":
                cin, h, w = layer["in_shape"]
                k = layer["k"]
                dcols, Ecols = dx, Ex
                dx = O.col2im(dcols, cin, batch, h, w, k)
                Ex = O.col2im(Ecols, cin, batch, h, w, k) + gamma(k * k) * O.col2im(
                    np.abs(dcols) + Ecols, cin, batch, h, w, k)
            d, E = dx, Ex
        elif kind == "pool2":
            cs, b, h, w = c["shape"]
            d = O.maxpool2_bwd(d.reshape(cs, b, h // 2, w // 2), c["idx"])
            E = O.maxpool2_bwd(E.reshape(cs, b, h // 2, w // 2), c["idx"])
        elif kind == "flatten":
            cs, b, h, w = c["shape"]
            d, E = O.unflatten_cnhw(d, cs, b, h, w), O.unflatten_cnhw(E, cs, b, h, w)
    return out


def assert_within(got, ref, limit, rtol=1e-4, atol=1e-6, what=""):
    """Every element passes |got - ref| <= atol + rtol |ref| or, failing that,
    the carried bound ``limit``. Returns how many needed the bound."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    err = np.abs(got - ref)
    first = err <= atol + rtol * np.abs(ref)
    second = err <= np.asarray(limit, dtype=np.float64) * (1.0 + 1e-6) + 1e-30
    bad = ~(first | second)
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{what}: {int(bad.sum())} entries beyond the carried bound, e.g. "
                             f"{[(tuple(i), got[tuple(i)], ref[tuple(i)], float(np.asarray(limit)[tuple(i)])) for i in idx]}")
    return int((~first).sum())
