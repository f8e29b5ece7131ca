"""Pins of the CPU oracle against facts fixed outside the oracle itself.

Each test checks the oracle against something the paper prints, a closed
form, a textbook definition written as an independent loop, an invariant the
paper states, or finite differences. None of them re-types the oracle's own
formula.
"""

import json
import os

import numpy as np
import pytest

import oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")
F32 = np.float32


def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _rand_sparse(rng, m, k, density, dtype=F32):
    w = rng.standard_normal((m, k)) * (rng.random((m, k)) < density)
    return w.astype(dtype)


# --- worked example, Section 3.1 Figure "spformats" -------------------------

def test_csr_worked_example_bit_exact():
    d = _load("csr_worked_example.json")
    a = np.array(d["dense"], dtype=F32)
    w = O.csr_from_dense(a)
    assert w.row_ptr.tolist() == d["row_ptrs"]
    assert w.col_idx.tolist() == d["col_indices"]
    assert w.val.tolist() == d["elements"]
    np.testing.assert_array_equal(O.csr_to_dense(w), a)


def test_worked_example_products_and_transpose():
    d = _load("csr_worked_example.json")
    h = d["hand_derived"]
    w = O.csr_from_dense(np.array(d["dense"], dtype=F32))
    ones = np.ones((4, 1))
    assert O.spmm_fwd(w, ones)[:, 0].tolist() == h["A_times_ones"]
    assert O.spmm_bwd_t(w, ones)[:, 0].tolist() == h["At_times_ones"]
    trp, tci, tv, tpos = O.csr_transpose(w)
    assert trp.tolist() == h["transpose_row_ptrs"]
    assert tci.tolist() == h["transpose_col_indices"]
    assert tv.tolist() == h["transpose_elements"]
    assert tpos.tolist() == h["transpose_pos_of_each_csr_entry"]


# --- CSR construction and transposition ------------------------------------

@pytest.mark.parametrize("m,k,density", [(1, 1, 1.0), (5, 7, 0.3), (16, 3, 0.0),
                                         (9, 16, 1.0), (13, 11, 0.5)])
def test_csr_roundtrip_and_transpose_definition(m, k, density):
    rng = np.random.default_rng(m * 100 + k)
    a = _rand_sparse(rng, m, k, density)
    a[0, :] = 0.0                                   # an empty row
    w = O.csr_from_dense(a)
    # brute force: nnz, per-row counts, ascending columns
    assert w.nnz == int((a != 0).sum())
    for i in range(m):
        s, e = w.row_ptr[i], w.row_ptr[i + 1]
        cols = w.col_idx[s:e].tolist()
        assert cols == [j for j in range(k) if a[i, j] != 0]
    np.testing.assert_array_equal(O.csr_to_dense(w), a)
    trp, tci, tv, tpos = O.csr_transpose(w)
    wt = O.csr_from_dense(a.T.copy())
    np.testing.assert_array_equal(trp, wt.row_ptr)
    np.testing.assert_array_equal(tci, wt.col_idx)
    np.testing.assert_array_equal(tv, wt.val)
    np.testing.assert_array_equal(tv[tpos], w.val)


def test_negative_zero_dropped_nan_kept():
    a = np.array([[-0.0, 1.0, np.nan, 0.0]], dtype=F32)
    w = O.csr_from_dense(a)
    assert w.col_idx.tolist() == [1, 2]


# --- products: dense brute force and the paper's orientation -----------------

@pytest.mark.parametrize("m,k,n,density", [(6, 5, 3, 0.5), (16, 16, 1, 0.2),
                                           (3, 9, 7, 1.0), (8, 4, 5, 0.0)])
def test_spmm_against_dense_triple_loop(m, k, n, density):
    rng = np.random.default_rng(7 + m + k + n)
    a = _rand_sparse(rng, m, k, density)
    a[m // 2, :] = 0.0
    w = O.csr_from_dense(a)
    x = rng.standard_normal((k, n))
    dy = rng.standard_normal((m, n))
    y_loop = np.zeros((m, n))
    dx_loop = np.zeros((k, n))
    g_loop = np.zeros((m, k))
    for i in range(m):
        for j in range(k):
            for c in range(n):
                y_loop[i, c] += float(a[i, j]) * x[j, c]
                dx_loop[j, c] += float(a[i, j]) * dy[i, c]
                g_loop[i, j] += dy[i, c] * x[j, c]
    np.testing.assert_allclose(O.spmm_fwd(w, x), y_loop, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(O.spmm_bwd_t(w, dy), dx_loop, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(O.weight_grad_dense(dy, x), g_loop, rtol=1e-12, atol=1e-12)
    rows = w.row_of_each_entry()
    np.testing.assert_allclose(O.weight_grad_sddmm(w, dy, x),
                               g_loop[rows, w.col_idx], rtol=1e-12, atol=1e-12)


def test_forward_backward_match_paper_orientation():
    # Section 3.2: Forward X_T = X_B W', Backward dX_B = dX_T W (samples in rows)
    rng = np.random.default_rng(3)
    a = _rand_sparse(rng, 7, 6, 0.4)
    a[2, :] = 0.0                                  # empty row
    w = O.csr_from_dense(a)
    xb = rng.standard_normal((4, 6))              # 4 samples x 6 inputs
    dxt = rng.standard_normal((4, 7))
    np.testing.assert_allclose(O.dense_times_compressed_t(xb, w), O.spmm_fwd(w, xb.T).T,
                               rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(O.dense_times_compressed(dxt, w), O.spmm_bwd_t(w, dxt.T).T,
                               rtol=1e-12, atol=1e-12)


# --- prox: Section 2.2 closed form vs Section 3.3 min/max kernel form --------

def test_prox_hand_cases():
    d = _load("soft_threshold_cases.json")
    ws = np.array([[c["w"] for c in d["cases"]]], dtype=F32)
    gs = np.array([[c["g"] for c in d["cases"]]], dtype=F32)
    w = O.csr_from_dense(ws)
    out = O.prox_update_compact(w, gs, d["eta"], d["lambda"])
    dense = O.csr_to_dense(out)[0]
    for j, c in enumerate(d["cases"]):
        assert (dense[j] != 0) == c["kept"], c
        assert dense[j] == F32(c["out"]), c
    assert out.nnz == sum(c["kept"] for c in d["cases"])


def _minmax_form(z, thr):
    # Section 3.3 kernel: A <- min(max(A - thr, 0), A + thr), evaluated in float32
    return np.minimum(np.maximum(z - thr, F32(0)), z + thr).astype(F32)


def test_prox_closed_form_equals_kernel_form_bitwise():
    rng = np.random.default_rng(11)
    for eta, lam in [(0.01, 1e-4), (0.5, 0.25), (1e-3, 3.0), (0.1, 0.0)]:
        m, k = 37, 53
        a = _rand_sparse(rng, m, k, 0.3)
        g = rng.standard_normal((m, k)).astype(F32) * F32(10 ** rng.uniform(-6, 2))
        w = O.csr_from_dense(a)
        out = O.csr_to_dense(O.prox_update_compact(w, g, eta, lam))
        thr = F32(eta) * F32(lam)
        z = a - F32(eta) * g
        ref = _minmax_form(z, thr)
        ref[ref == 0] = 0.0                        # -0.0 from min(.,.) is "not stored"
        np.testing.assert_array_equal(out.view(np.uint32), ref.view(np.uint32))


def test_prox_identity_empty_and_nesting():
    rng = np.random.default_rng(5)
    a = _rand_sparse(rng, 20, 30, 0.25)
    a[3, 4] = 0.0
    w = O.csr_from_dense(a)
    zero_g = np.zeros_like(a)
    same = O.prox_update_compact(w, zero_g, 0.1, 0.0)     # G = 0, lambda = 0
    np.testing.assert_array_equal(O.csr_to_dense(same), a)
    assert same.nnz == w.nnz
    g = rng.standard_normal(a.shape).astype(F32)
    empty = O.prox_update_compact(w, g, 0.1, 1e30)
    assert empty.nnz == 0 and empty.row_ptr.tolist() == [0] * 21
    prev = None
    for lam in [0.0, 1e-3, 1e-2, 0.1, 1.0, 10.0]:
        pat = O.csr_to_dense(O.prox_update_compact(w, g, 0.1, lam)) != 0
        if prev is not None:
            assert not (pat & ~prev).any()          # larger lambda: a subset
        prev = pat


def test_prox_reentry_of_zero_weights():
    # Section 3.3 applies the prox to the dense w - eta*G: an off-pattern entry
    # with |eta*g| > eta*lambda enters the pattern.
    w = O.csr_from_dense(np.zeros((1, 3), dtype=F32))
    g = np.array([[1.0, -1.0, 1e-6]], dtype=F32)
    out = O.prox_update_compact(w, g, 0.5, 0.25)
    assert out.col_idx.tolist() == [0, 1]
    assert out.val.tolist() == [-0.375, 0.375]


def test_debias_keeps_pattern():
    rng = np.random.default_rng(8)
    a = _rand_sparse(rng, 12, 9, 0.4)
    w = O.csr_from_dense(a)
    g = rng.standard_normal(w.nnz).astype(F32)
    g[0] = w.val[0] / F32(0.5)                    # drives entry 0 exactly to zero
    out = O.debias_update(w, g, 0.5)
    np.testing.assert_array_equal(out.row_ptr, w.row_ptr)
    np.testing.assert_array_equal(out.col_idx, w.col_idx)
    assert out.val[0] == 0.0                       # stays stored
    np.testing.assert_array_equal(out.val[1:], (w.val[1:] - F32(0.5) * g[1:]).astype(F32))


# --- glue layers against direct definitions ---------------------------------

def test_im2col_matches_direct_convolution_and_col2im_is_adjoint():
    rng = np.random.default_rng(2)
    c, b, h, wd, k, cout = 2, 3, 6, 5, 3, 4
    x = rng.standard_normal((c, b, h, wd))
    wt = rng.standard_normal((cout, c * k * k))
    y = (wt @ O.im2col(x, k)).reshape(cout, b, h - k + 1, wd - k + 1)
    ref = np.zeros_like(y)
    for o in range(cout):
        for bb in range(b):
            for oy in range(h - k + 1):
                for ox in range(wd - k + 1):
                    s = 0.0
                    for ci in range(c):
                        for ky in range(k):
                            for kx in range(k):
                                s += wt[o, ci * k * k + ky * k + kx] * x[ci, bb, oy + ky, ox + kx]
                    ref[o, bb, oy, ox] = s
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)
    cols = rng.standard_normal((c * k * k, b * (h - k + 1) * (wd - k + 1)))
    lhs = np.sum(O.im2col(x, k) * cols)
    rhs = np.sum(x * O.col2im(cols, c, b, h, wd, k))
    assert abs(lhs - rhs) < 1e-9 * max(1.0, abs(lhs))


def test_maxpool_against_loops_with_ties():
    x = np.array([[[[1, 3, 2, 2], [3, 0, 2, 2], [-1, -2, 5, 4], [-3, -1, 4, 5]]]], dtype=float)
    y, idx = O.maxpool2_fwd(x)
    assert y[0, 0].tolist() == [[3, 2], [-1, 5]]
    assert idx[0, 0].tolist() == [[1, 0], [0, 0]]  # first maximum in scan order wins
    dx = O.maxpool2_bwd(np.ones((1, 1, 2, 2)), idx)
    assert dx[0, 0].tolist() == [[0, 1, 1, 0], [0, 0, 0, 0], [1, 0, 1, 0], [0, 0, 0, 0]]


def test_softmax_xent_closed_forms():
    z = np.zeros((10, 4))
    loss, dz = O.softmax_xent(z, np.array([0, 3, 9, 9]))
    assert abs(loss - np.log(10)) < 1e-15
    np.testing.assert_allclose(dz.sum(axis=0), 0, atol=1e-15)
    assert abs(dz[3, 1] - (0.1 - 1) / 4) < 1e-15


def test_flatten_is_caffe_order():
    x = np.arange(2 * 3 * 2 * 2).reshape(2, 3, 2, 2)   # (C, B, h, w)
    xf = O.flatten_cnhw(x)
    for c in range(2):
        for b in range(3):
            for yy in range(2):
                for xx in range(2):
                    assert xf[c * 4 + yy * 2 + xx, b] == x[c, b, yy, xx]
    np.testing.assert_array_equal(O.unflatten_cnhw(xf, 2, 3, 2, 2), x)


# --- finite differences of the whole step -----------------------------------

def _fd_check(net, dense_ws, biases, x0, labels, h=1e-5, rtol=1e-5):
    params = []
    wi = 0
    for layer in net.layers:
        if layer["kind"] in ("fc", "conv"):
            params.append({"W": O.csr_from_dense(dense_ws[wi]), "b": biases[wi]})
            wi += 1
        else:
            params.append(None)
    net.params = params
    logits, cache = O.net_forward(net, x0, len(labels))
    _, dz = O.softmax_xent(logits, labels)
    gp = O.net_backward(net, cache, dz, "prox")
    gd = O.net_backward(net, cache, dz, "debias")
    pl = [i for i, l in enumerate(net.layers) if l["kind"] in ("fc", "conv")]
    rng = np.random.default_rng(1)
    for wi, li in enumerate(pl):
        a = dense_ws[wi]
        stored = list(zip(*np.nonzero(a != 0)))
        zeros = list(zip(*np.nonzero(a == 0)))
        picks = [stored[t] for t in rng.choice(len(stored), min(4, len(stored)), replace=False)]
        picks += [zeros[t] for t in rng.choice(len(zeros), min(4, len(zeros)), replace=False)]
        for (i, j) in picks:
            wp = [w.copy() for w in dense_ws]
            wm = [w.copy() for w in dense_ws]
            wp[wi][i, j] += h
            wm[wi][i, j] -= h
            fd = (O.net_loss_dense(net, wp, biases, x0, labels)
                  - O.net_loss_dense(net, wm, biases, x0, labels)) / (2 * h)
            an = gp[li]["G"][i, j]
            assert abs(fd - an) <= rtol * max(abs(fd), 1e-3), (li, i, j, fd, an)
            if a[i, j] != 0:
                w = net.params[li]["W"]
                k = int(w.row_ptr[i]) + int(np.searchsorted(
                    w.col_idx[w.row_ptr[i]:w.row_ptr[i + 1]], j))
                assert abs(gd[li]["g"][k] - an) <= 1e-12 * max(1.0, abs(an))
        for i in range(min(3, len(biases[wi]))):
            bp = [b.copy() for b in biases]
            bm = [b.copy() for b in biases]
            bp[wi][i] += h
            bm[wi][i] -= h
            fd = (O.net_loss_dense(net, dense_ws, bp, x0, labels)
                  - O.net_loss_dense(net, dense_ws, bm, x0, labels)) / (2 * h)
            assert abs(fd - gp[li]["gb"][i]) <= rtol * max(abs(fd), 1e-3)


def test_finite_differences_tiny_mlp():
    rng = np.random.default_rng(4)
    sizes = [6, 5, 4, 3]
    ws = [rng.standard_normal((m, k)) * (rng.random((m, k)) < 0.6)
          for k, m in zip(sizes[:-1], sizes[1:])]
    bs = [rng.standard_normal(m) * 0.1 for m in sizes[1:]]
    net = O.Net([{"kind": "fc", "relu": True}, {"kind": "fc", "relu": True},
                 {"kind": "fc", "relu": False}])
    x = rng.standard_normal((6, 3))
    _fd_check(net, ws, bs, x, np.array([0, 2, 1]))


def test_finite_differences_tiny_conv_net():
    rng = np.random.default_rng(6)
    # conv 3x(1*3*3) on 1x8x8 -> 3x6x6, pool -> 3x3x3? use 10x10 -> 8x8 -> 4x4
    # conv 2x(3*3*3) -> 2x2x2, pool -> 2x1x1, flatten 2, fc 2->3
    layers = [{"kind": "conv", "k": 3, "in_shape": (1, 10, 10), "relu": False},
              {"kind": "pool2"},
              {"kind": "conv", "k": 3, "in_shape": (3, 4, 4), "relu": False},
              {"kind": "pool2"},
              {"kind": "flatten"},
              {"kind": "fc", "relu": True},
              {"kind": "fc", "relu": False}]
    ws = [rng.standard_normal((3, 9)) * (rng.random((3, 9)) < 0.7),
          rng.standard_normal((2, 27)) * (rng.random((2, 27)) < 0.7),
          rng.standard_normal((4, 2)),
          rng.standard_normal((3, 4)) * (rng.random((3, 4)) < 0.7)]
    bs = [rng.standard_normal(3) * 0.1, rng.standard_normal(2) * 0.1,
          rng.standard_normal(4) * 0.1, rng.standard_normal(3) * 0.1]
    x = rng.standard_normal((1, 2, 10, 10))
    _fd_check(O.Net(layers), ws, bs, x, np.array([1, 2]))


# --- a planted mistake must fail a pin (the mistake lives here, on the CPU) --

def test_pins_catch_a_transposed_operand():
    d = _load("csr_worked_example.json")
    w = O.csr_from_dense(np.array(d["dense"], dtype=F32))
    wrong = O.spmm_fwd(w, np.ones((4, 1)))[:, 0].tolist()   # W instead of W^T
    assert wrong != d["hand_derived"]["At_times_ones"]


def test_pins_catch_a_wrong_threshold_sign():
    d = _load("soft_threshold_cases.json")
    c = d["cases"][3]                               # z = -1.25
    thr = F32(d["eta"]) * F32(d["lambda"])
    z = F32(c["w"]) - F32(d["eta"]) * F32(c["g"])
    assert F32(z - thr) != F32(c["out"])            # sign mistake is caught


# --- Prox-RMSProp (Algorithm 1) and Prox-ADAM (Algorithm 2) -----------------

def _one_entry(w):
    return O.csr_from_dense(np.array([[w]], dtype=F32))


def _dense_value(csr):
    return None if csr.nnz == 0 else float(O.csr_to_dense(csr)[0, 0])


def test_rmsprop_hand_cases():
    d = _load("adaptive_prox_cases.json")
    for c in d["rmsprop"]:
        g = np.array([[c["g"]]], dtype=F32)
        v = np.array([[c["v"]]], dtype=F32)
        v_new, dd = O.rmsprop_direction(g, v, c["beta"], c["eps"])
        assert v_new[0, 0] == F32(c["v_new"]) and dd[0, 0] == F32(c["d"]), c
        w_new, v2 = O.prox_rmsprop_update_compact(_one_entry(c["w"]), g, v, d["eta"], d["lambda"], c["beta"],
                                                  c["eps"])
        assert _dense_value(w_new) == c["w_new"], c
        assert v2[0, 0] == F32(c["v_new"])


def test_adam_hand_cases():
    d = _load("adaptive_prox_cases.json")
    for c in d["adam"]:
        g = np.array([[c["g"]]], dtype=F32)
        m = np.array([[c["m"]]], dtype=F32)
        v = np.array([[c["v"]]], dtype=F32)
        m_new, v_new, dd = O.adam_direction(g, m, v, c["t"], c["beta1"], c["beta2"], c["eps"])
        assert (m_new[0, 0], v_new[0, 0], dd[0, 0]) == (F32(c["m_new"]), F32(c["v_new"]), F32(c["d"])), c
        w_new, m2, v2 = O.prox_adam_update_compact(_one_entry(c["w"]), g, m, v, c["t"], d["eta"], d["lambda"],
                                                   c["beta1"], c["beta2"], c["eps"])
        assert _dense_value(w_new) == c["w_new"], c
        assert m2[0, 0] == F32(c["m_new"]) and v2[0, 0] == F32(c["v_new"])


def test_adam_without_momentum_is_rmsprop_without_averaging():
    # beta1 = beta2 = 0: m_hat = g and v_hat = g*g, the bias corrections are 1;
    # RMSProp with beta = 0 has v = g*g: the two directions agree bit for bit.
    rng = np.random.default_rng(5)
    g = rng.standard_normal((7, 9)).astype(F32)
    m = rng.standard_normal((7, 9)).astype(F32)
    v = np.abs(rng.standard_normal((7, 9))).astype(F32)
    _, _, d_adam = O.adam_direction(g, m, v, 3, 0.0, 0.0, 1e-3)
    _, d_rms = O.rmsprop_direction(g, v, 0.0, 1e-3)
    np.testing.assert_array_equal(d_adam.view(np.uint32), d_rms.view(np.uint32))


def _textbook_adam(w, gs, eta, b1, b2, eps):
    m = np.zeros_like(w)
    v = np.zeros_like(w)
    for t, g in enumerate(gs, start=1):
        m = b1 * m + (1 - b1) * g
        v = b2 * v + (1 - b2) * g * g
        w = w - eta * (m / (1 - b1 ** t)) / (np.sqrt(v / (1 - b2 ** t)) + eps)
    return w


def _textbook_rmsprop(w, gs, eta, beta, eps):
    v = np.zeros_like(w)
    for g in gs:
        v = beta * v + (1 - beta) * g * g
        w = w - eta * g / (np.sqrt(v) + eps)
    return w


def test_adaptive_trajectories_match_textbook_float64():
    # lambda = 0: the prox is the identity (only exact zeros drop), so five
    # steps must follow the float64 textbook method within float32 rounding
    rng = np.random.default_rng(21)
    w0 = rng.standard_normal((6, 10)).astype(F32)
    gs = [rng.standard_normal((6, 10)).astype(F32) for _ in range(5)]
    eta, b1, b2, eps = 0.01, 0.9, 0.999, 1e-8
    w = O.csr_from_dense(w0)
    m = np.zeros_like(w0)
    v = np.zeros_like(w0)
    for t, g in enumerate(gs, start=1):
        w, m, v = O.prox_adam_update_compact(w, g, m, v, t, eta, 0.0, b1, b2, eps)
    ref = _textbook_adam(w0.astype(np.float64), [g.astype(np.float64) for g in gs], eta, b1, b2, eps)
    np.testing.assert_allclose(O.csr_to_dense(w), ref, rtol=0, atol=2e-6)
    w = O.csr_from_dense(w0)
    v = np.zeros_like(w0)
    for g in gs:
        w, v = O.prox_rmsprop_update_compact(w, g, v, eta, 0.0, 0.9, eps)
    ref = _textbook_rmsprop(w0.astype(np.float64), [g.astype(np.float64) for g in gs], eta, 0.9, eps)
    np.testing.assert_allclose(O.csr_to_dense(w), ref, rtol=0, atol=2e-6)


def test_adaptive_threshold_is_eta_lambda():
    # the threshold is eta*lambda, not divided by the adaptive denominator:
    # Adam's first step moves every entry by about eta (|d| ~ 1), so with
    # eta*lambda above eta everything starting at 0 is dropped, and below it
    # everything is kept
    rng = np.random.default_rng(8)
    g = rng.standard_normal((5, 8)).astype(F32)
    zero = O.csr_from_dense(np.zeros((5, 8), dtype=F32))
    z = np.zeros((5, 8), dtype=F32)
    w_big, _, _ = O.prox_adam_update_compact(zero, g, z, z, 1, 0.1, 1.5, 0.9, 0.999, 1e-8)
    w_small, _, _ = O.prox_adam_update_compact(zero, g, z, z, 1, 0.1, 0.5, 0.9, 0.999, 1e-8)
    assert w_big.nnz == 0 and w_small.nnz == 40


def test_pins_catch_a_missing_bias_correction():
    d = _load("adaptive_prox_cases.json")
    c = d["adam"][0]
    c1, c2 = F32(1) - F32(c["beta1"]), F32(1) - F32(c["beta2"])
    m_new = c1 * F32(c["g"])
    v_new = c2 * F32(c["g"]) * F32(c["g"])
    wrong = m_new / (np.sqrt(v_new) + F32(c["eps"]))          # no division by 1 - beta^t
    assert F32(wrong) != F32(c["d"])


def test_pins_catch_the_old_second_moment():
    d = _load("adaptive_prox_cases.json")
    c = d["rmsprop"][0]
    wrong = F32(c["g"]) / (np.sqrt(F32(c["v"])) + F32(c["eps"]))   # v_{t-1} instead of v_t
    assert F32(wrong) != F32(c["d"])
