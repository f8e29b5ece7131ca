"""The carried element-wise bound of tests/chain_bound.py, checked on the CPU.

A float32 evaluation of the same network (numpy float32 products, whose
summation order is numpy's, not CSR order) must lie inside the bound at every
element of the logits and of every layer's dL/dpre; the bound must be tight
enough to mean something (a worst-case bound widens by the cancellation
factor sum |terms| / |sum| at every layer it crosses: its median relative
width stays below 1%, far below the max-norm test it replaces for small
entries); and an error planted in one element of the float32 chain (a
dropped term) must be caught.
"""

import numpy as np
import pytest

import oracle as O
from tests import chain_bound

F32 = np.float32


def _net(rng, sizes, densities):
    layers = [{"kind": "fc", "relu": i < len(sizes) - 2} for i in range(len(sizes) - 1)]
    params, dense = [], []
    for (k, m), d in zip(zip(sizes[:-1], sizes[1:]), densities):
        w = np.where(rng.random((m, k)) < d, rng.normal(0, np.sqrt(2.0 / k), (m, k)), 0).astype(F32)
        b = rng.normal(0, 0.1, m).astype(F32)
        dense.append(w)
        params.append({"W": O.csr_from_dense(w), "b": b})
    return O.Net(layers, params), dense


def _float32_chain(net, dense, x, labels):
    """Forward and backward of an fc net in float32 (numpy's summation order)."""
    ys, pres = [x.astype(F32)], []
    for layer, p, w in zip(net.layers, net.params, dense):
        pre = (w @ ys[-1] + p["b"][:, None]).astype(F32)
        pres.append(pre)
        ys.append(np.maximum(pre, F32(0)) if layer["relu"] else pre)
    z = ys[-1]
    e = np.exp(z - z.max(axis=0, keepdims=True)).astype(F32)
    p = (e / e.sum(axis=0, keepdims=True)).astype(F32)
    n = z.shape[1]
    d = p.copy()
    d[labels, np.arange(n)] -= F32(1)
    d = (d / F32(n)).astype(F32)
    deltas = [None] * len(dense)
    for li in range(len(dense) - 1, -1, -1):
        if net.layers[li]["relu"]:
            d = np.where(pres[li] > 0, d, F32(0)).astype(F32)
        deltas[li] = d
        d = (dense[li].T @ d).astype(F32)
    return z, deltas


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_float32_chain_lies_inside_the_bound(seed):
    rng = np.random.default_rng(seed)
    net, dense = _net(rng, (300, 200, 100, 10), (0.3, 0.2, 0.5))
    n = 64
    x = rng.random((300, n)).astype(F32)
    labels = rng.integers(0, 10, n)
    z32, d32 = _float32_chain(net, dense, x, labels)
    logits, F, per = chain_bound.forward_bounds(net, x, n)
    chain_bound.assert_within(z32, logits, F, rtol=0, atol=0, what="logits")
    dz, E = chain_bound.softmax_bound(logits, F, labels)
    back = chain_bound.backward_bounds(net, per, dz, E, n)
    for li in range(3):
        ref, lim = back[li]
        chain_bound.assert_within(d32[li], ref, lim, rtol=0, atol=0, what=f"delta {li}")
        live = np.abs(ref) > 1e-3 * np.abs(ref).max()
        assert np.median(lim[live] / np.abs(ref[live])) < 1e-2, "bound too loose to mean anything"


def test_planted_dropped_term_is_caught():
    rng = np.random.default_rng(5)
    net, dense = _net(rng, (300, 200, 100, 10), (0.3, 0.2, 0.5))
    n = 32
    x = rng.random((300, n)).astype(F32)
    labels = rng.integers(0, 10, n)
    # drop one stored term of the middle layer's product in the float32 chain
    w_bad = [w.copy() for w in dense]
    r, c = np.argwhere(w_bad[1] != 0)[7]
    w_bad[1][r, c] = 0
    _, d32 = _float32_chain(net, w_bad, x, labels)
    logits, F, per = chain_bound.forward_bounds(net, x, n)
    dz, E = chain_bound.softmax_bound(logits, F, labels)
    back = chain_bound.backward_bounds(net, per, dz, E, n)
    with pytest.raises(AssertionError):
        for li in range(3):
            chain_bound.assert_within(d32[li], back[li][0], back[li][1], rtol=0, atol=0, what=f"delta {li}")


def test_conv_chain_bound_covers_a_float32_lenet_forward():
    """im2col, pooling and flatten carry the bound: a float32 forward of a
    small conv net (products in numpy float32) lies inside it."""
    rng = np.random.default_rng(3)
    layers = [{"kind": "conv", "k": 3, "in_shape": (2, 10, 10), "relu": False}, {"kind": "pool2"},
              {"kind": "flatten"}, {"kind": "fc", "relu": True}, {"kind": "fc", "relu": False}]
    shapes = [(4, 18), (12, 64), (5, 12)]
    dense = [np.where(rng.random(s) < 0.5, rng.normal(0, 0.5, s), 0).astype(F32) for s in shapes]
    bs = [rng.normal(0, 0.1, s[0]).astype(F32) for s in shapes]
    params, wi = [], 0
    for L in layers:
        if L["kind"] in ("fc", "conv"):
            params.append({"W": O.csr_from_dense(dense[wi]), "b": bs[wi]})
            wi += 1
        else:
            params.append(None)
    net = O.Net(layers, params)
    b = 6
    x = rng.random((2, b, 10, 10)).astype(F32)
    cols = O.im2col(x, 3).astype(F32)
    y = (dense[0] @ cols + bs[0][:, None]).astype(F32).reshape(4, b, 8, 8)
    yp, _ = O.maxpool2_fwd(y)
    f = O.flatten_cnhw(yp).astype(F32)
    h = np.maximum((dense[1] @ f + bs[1][:, None]).astype(F32), F32(0))
    z32 = (dense[2] @ h + bs[2][:, None]).astype(F32)
    logits, F, _ = chain_bound.forward_bounds(net, x, b)
    chain_bound.assert_within(z32, logits, F, rtol=0, atol=0, what="conv logits")
