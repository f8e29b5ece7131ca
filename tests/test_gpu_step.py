"""Whole training steps of the five workloads against the oracle.

Each GPU step is compared with the oracle run on the same current weights:
the loss, every layer's gradient (dense G in the prox phase, g at the stored
entries in the debias phase), and the updated CSR, which must be bit-exact
with the oracle's update re-fed the GPU's own gradient (the gradients agree
only up to summation order, so a free-running pattern could differ where
|w - eta*G| sits within rounding of eta*lambda).
"""

import numpy as np
import pytest

import oracle as O
from tests import chain_bound
from tests.parity import assert_close, csr_dense

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu
F32 = np.float32


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import csrtrain
    csrtrain.lib()
    return csrtrain


def _host_csr(w):
    (rp, ci, v), t = w.to_host()
    return O.CSR(w.rows, w.cols, rp.copy(), ci.copy(), v.copy()), t


def _assert_csr_bits(w, ref):
    got, t = _host_csr(w)
    np.testing.assert_array_equal(got.row_ptr, ref.row_ptr)
    np.testing.assert_array_equal(got.col_idx, ref.col_idx)
    np.testing.assert_array_equal(got.val.view(np.uint32), ref.val.astype(F32).view(np.uint32))
    if t is not None:
        trp, tci, tv, tpos = O.csr_transpose(ref)
        np.testing.assert_array_equal(t[0], trp)
        np.testing.assert_array_equal(t[1], tci)
        np.testing.assert_array_equal(t[2].view(np.uint32), tv.astype(F32).view(np.uint32))
        np.testing.assert_array_equal(t[3], tpos)


@pytest.mark.parametrize("prec", [0, 1])
def test_single_fc_layer_step(C, prec):
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SingleLayer
    cfg = synth.single_fc(seed=0)
    lay = SingleLayer(cfg["W"], cfg["X"].shape[1], precision=prec)
    lay.x.copy_(torch.from_numpy(cfg["X"]))
    lay.dy.copy_(torch.from_numpy(cfg["dY"]))
    w0 = O.csr_from_dense(cfg["W"])
    _assert_csr_bits(lay.W[0], w0)
    lay.step(cfg["eta"], cfg["lambda"])
    torch.cuda.synchronize()
    x, dy = cfg["X"], cfg["dY"]
    assert_close(lay.y.cpu().numpy(), O.spmm_fwd(w0, x), O.spmm_fwd(O.csr_abs(w0), np.abs(x)),
                 np.diff(w0.row_ptr)[:, None], what="Y")
    assert_close(lay.dx.cpu().numpy(), O.spmm_bwd_t(w0, dy), O.spmm_bwd_t(O.csr_abs(w0), np.abs(dy)),
                 np.bincount(w0.col_idx, minlength=w0.cols)[:, None], what="dX")
    G = lay.G.cpu().numpy()
    assert_close(G, O.weight_grad_dense(dy, x), O.weight_grad_dense(np.abs(dy), np.abs(x)), x.shape[1],
                 rtol=1e-3 if prec else 1e-4, tf32=bool(prec), what="G")
    _assert_csr_bits(lay.W[1], O.prox_update_compact(w0, G, cfg["eta"], cfg["lambda"]))
    nnz = lay.W[1].nnz()
    assert nnz > w0.nnz                                 # zero weights re-enter (dense w - eta*G)


def _oracle_net(layers, net):
    onet = O.Net([dict(l) for l in layers], [])
    pi = 0
    for L in layers:
        if L["kind"] in ("fc", "conv"):
            w, _ = _host_csr(net.weights(pi))
            onet.params.append({"W": w, "b": net.params[pi]["b"].cpu().numpy().copy()})
            pi += 1
        else:
            onet.params.append(None)
    return onet


def _run_and_compare(C, net, layers, x_host, labels, eta, lam, phase, prec):
    """One GPU step, checked against the oracle element by element.

    Each layer on the GPU's own inputs: its forward output against the oracle
    product of the GPU's layer input, dL/dpre of a layer below an fc layer
    against the oracle's transposed product of the GPU's dL/dpre above, its
    gradient against the oracle fed the GPU's dL/dpre and layer input, and the
    update bit for bit against the oracle update fed the GPU's gradient. The
    chain as a whole against the oracle's own float64 forward / backward: the
    loss, max-pool winners (exact except at near-ties, where either winner is
    correct) and every element of every layer's dL/dpre, within the error
    bound carried through the chain (tests/chain_bound.py).
    """
    onet = _oracle_net(layers, net)
    batch = len(labels)
    loss = net.step(phase, eta, lam)
    torch.cuda.synchronize()
    assert net.ws.status()[0] == 0
    logits, cache = O.net_forward(onet, x_host, batch)
    pool_idx = {}
    for li, L in enumerate(layers):
        if L["kind"] == "pool2":
            gidx = net.layers[li]["idx"].cpu().numpy().reshape(cache[li]["idx"].shape)
            diff = gidx != cache[li]["idx"]
            if diff.any():
                c, b, h, w = cache[li]["shape"]
                xin = net.layers[li]["x"].cpu().numpy().reshape(c, b, h, w).astype(np.float64)
                win = xin.reshape(c, b, h // 2, 2, w // 2, 2).transpose(0, 1, 2, 4, 3, 5).reshape(
                    c, b, h // 2, w // 2, 4)
                picked = np.take_along_axis(win, gidx[..., None].astype(np.int64), axis=-1)[..., 0]
                best = win.max(axis=-1)
                assert np.all(picked[diff] >= best[diff]), "GPU pooling picked a non-maximum"
                assert diff.mean() < 1e-3, diff.mean()
            pool_idx[li] = gidx.astype(np.int8)
    oloss, _ = O.softmax_xent(logits, labels)
    got_loss = float(loss[0].item())
    assert abs(got_loss - oloss) <= 2e-5 * max(1.0, abs(oloss)), (got_loss, oloss)
    # the chain: oracle forward / backward with carried element-wise bounds
    blogits, F_logits, per = chain_bound.forward_bounds(onet, x_host, batch, pool_idx)
    dz, E_dz = chain_bound.softmax_bound(blogits, F_logits, labels)
    chain = chain_bound.backward_bounds(onet, per, dz, E_dz, batch)
    pl = [i for i, l in enumerate(layers) if l["kind"] in ("fc", "conv")]
    for pi, li in enumerate(pl):
        L = net.params[pi]
        old = onet.params[li]
        W = old["W"]
        M = W.rows
        d_gpu = L["dpre"].cpu().numpy().reshape(M, -1).astype(np.float64)
        x_gpu = L["xmat"].cpu().numpy().reshape(W.cols, -1).astype(np.float64)
        n = x_gpu.shape[1]
        absx, absd = np.abs(x_gpu), np.abs(d_gpu)
        # this layer's forward output from the GPU's own input (im2col columns for a conv layer)
        pre = O.spmm_fwd(W, x_gpu) + old["b"].astype(np.float64)[:, None]
        want = O.relu(pre) if layers[li]["relu"] else pre
        assert_close(L["y"].cpu().numpy().reshape(M, -1).astype(np.float64), want,
                     lambda: O.spmm_fwd(O.csr_abs(W), absx) + np.abs(old["b"]).astype(np.float64)[:, None],
                     np.diff(W.row_ptr)[:, None] + 1, what=f"forward of layer {pi}")
        # dL/dpre of this layer from the GPU's dL/dpre of the fc layer above
        if pi + 1 < len(pl) and layers[pl[pi + 1]]["kind"] == "fc" and pl[pi + 1] == li + 1:
            up = net.params[pi + 1]
            Wu = onet.params[li + 1]["W"]
            d_up = up["dpre"].cpu().numpy().reshape(Wu.rows, -1).astype(np.float64)
            mask = (L["y"].cpu().numpy() > 0) if layers[li]["relu"] else np.ones_like(d_gpu, dtype=bool)
            assert_close(d_gpu, O.spmm_bwd_t(Wu, d_up) * mask,
                         lambda: O.spmm_bwd_t(O.csr_abs(Wu), np.abs(d_up)) * mask,
                         np.bincount(Wu.col_idx, minlength=Wu.cols)[:, None], what=f"dL/dpre of layer {pi}")
        # ... and from the oracle's own chain, within the carried bound
        d_ref, E_ref = chain[li]
        chain_bound.assert_within(d_gpu, d_ref, E_ref, what=f"chain dL/dpre of layer {pi}")
        if phase == "prox":
            G = L["G"].cpu().numpy()
            assert_close(G, O.weight_grad_dense(d_gpu, x_gpu), O.weight_grad_dense(absd, absx), n,
                         rtol=1e-3 if prec else 1e-4, tf32=bool(prec), what=f"G layer {pi}")
            _assert_csr_bits(net.weights(pi), O.prox_update_compact(W, G, eta, lam))
        else:
            g = L["g"].cpu().numpy()[: W.nnz]
            assert_close(g, O.weight_grad_sddmm(W, d_gpu, x_gpu), O.weight_grad_sddmm(W, absd, absx), n,
                         what=f"g layer {pi}")
            _assert_csr_bits(net.weights(pi), O.debias_update(W, g, eta))
    return got_loss


@pytest.mark.parametrize("prec", [0, 1])
def test_mlp_prox_then_debias(C, prec):
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, mlp_layers
    cfg = synth.mlp(seed=0)
    layers = mlp_layers(3)
    net = SparseNet(layers, cfg["W"], cfg["b"], 256, (784,), precision=prec, grad_per_layer=True)
    net.x_in.copy_(torch.from_numpy(cfg["X"]))
    net.labels.copy_(torch.from_numpy(cfg["labels"]))
    for _ in range(3):
        _run_and_compare(C, net, layers, cfg["X"], cfg["labels"], cfg["eta"], cfg["lambda"], "prox", prec)
    for _ in range(3):
        _run_and_compare(C, net, layers, cfg["X"], cfg["labels"], cfg["eta"], cfg["lambda"], "debias", prec)


def test_lenet_prox_then_debias(C):
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, lenet_layers
    cfg = synth.lenet(seed=0)
    layers = lenet_layers()
    net = SparseNet(layers, cfg["W"], cfg["b"], 128, (1, 28, 28), precision=1, grad_per_layer=True)
    net.x_in.copy_(torch.from_numpy(cfg["X"].reshape(1, -1)))
    net.labels.copy_(torch.from_numpy(cfg["labels"]))
    for phase in ("prox", "prox", "debias", "debias"):
        _run_and_compare(C, net, layers, cfg["X"], cfg["labels"], cfg["eta"], cfg["lambda"], phase, 1)


def test_fc_head_full_size_step(C):
    """The AlexNet-sized head (9216-4096-4096-1000, batch 256) at full size:
    one prox step and one debias step, every layer checked."""
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, mlp_layers
    cfg = synth.fc_head(seed=0)
    layers = mlp_layers(3)
    net = SparseNet(layers, cfg["W"], cfg["b"], 256, (9216,), precision=1, grad_per_layer=True)
    net.x_in.copy_(torch.from_numpy(cfg["X"]))
    net.labels.copy_(torch.from_numpy(cfg["labels"]))
    _run_and_compare(C, net, layers, cfg["X"], cfg["labels"], cfg["eta"], cfg["lambda"], "prox", 1)
    net.reset_weights()
    _run_and_compare(C, net, layers, cfg["X"], cfg["labels"], cfg["eta"], cfg["lambda"], "debias", 1)


def _assert_prox_within_bound(w_gpu, W_old, d, x, eta, lam, what):
    """The fused prox step (G never written) against the oracle's fp64 G from
    the same dL/dpre and layer input. G_gpu is within the TF32 summation bound
    tol of G, so z = w - eta*G moves by at most dz = eta*tol plus the two fp32
    roundings: every entry with | |z| - thr | > dz must take the oracle's keep
    decision, and every kept value must be within dz of z - sign(z)*thr."""
    got, t = _host_csr(w_gpu)
    M, K = W_old.rows, W_old.cols
    n = x.shape[1]
    G = O.weight_grad_dense(d, x)
    S = O.weight_grad_dense(np.abs(d), np.abs(x))
    from tests.parity import TF32_OPERAND, U32, gamma
    tol = gamma(n + 1) * S + U32 * np.abs(G) + 2 * TF32_OPERAND * S + 1e-30
    w0 = csr_dense(W_old.row_ptr, W_old.col_idx, W_old.val, M, K).astype(np.float64)
    thr = float(np.float32(eta) * np.float32(lam))
    z = w0 - eta * G
    dz = 2.0 * (eta * tol + U32 * (eta * np.abs(G) + np.abs(z))) + 1e-30
    keep = np.zeros((M, K), dtype=bool)
    keep[np.repeat(np.arange(M), np.diff(got.row_ptr.astype(np.int64))), got.col_idx] = True
    clear = np.abs(np.abs(z) - thr) > dz
    wrong = clear & (keep != (np.abs(z) > thr))
    assert not wrong.any(), f"{what}: {int(wrong.sum())} keep decisions outside the bound"
    vg = csr_dense(got.row_ptr, got.col_idx, got.val, M, K).astype(np.float64)
    ref = z - np.sign(z) * thr
    err = np.abs(vg - ref)[keep]
    assert np.all(err <= dz[keep] + U32 * np.abs(ref[keep])), f"{what}: kept values beyond the bound"
    assert np.all(np.diff(got.row_ptr) >= 0) and got.row_ptr[0] == 0
    # columns strictly ascending within every row
    rp64 = got.row_ptr.astype(np.int64)
    if got.nnz > 1:
        step_up = np.diff(got.col_idx.astype(np.int64)) > 0
        row_start = np.zeros(got.nnz, dtype=bool)
        row_start[rp64[1:-1][rp64[1:-1] < got.nnz]] = True
        assert np.all(step_up | row_start[1:]), f"{what}: columns not strictly ascending within a row"
    if t is not None:   # the transposed copy is exactly the transpose of the GPU's own CSR
        trp, tci, tv, tpos = O.csr_transpose(got)
        np.testing.assert_array_equal(t[0], trp)
        np.testing.assert_array_equal(t[1], tci)
        np.testing.assert_array_equal(t[2].view(np.uint32), tv.astype(F32).view(np.uint32))
        np.testing.assert_array_equal(t[3], tpos)
    in_band = int((~clear).sum())
    print(f"{what}: {int(keep.sum())} kept, {in_band} of {M * K} entries inside the TF32 band")
    assert in_band <= 0.1 * M * K, f"{what}: {in_band} entries inside the band"
    return int(keep.sum()), in_band


@pytest.mark.parametrize("workload", ["mlp", "fc_head"])
def test_fused_prox_step(C, workload):
    """The network's default prox phase: weight gradient and prox update in
    one tensor-core pass per layer (shapes it does not cover take the
    unfused calls), checked against the oracle on the GPU's own dL/dpre."""
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, mlp_layers
    # 320-192-100-10: two layers fused, the last (K = 100) on the unfused calls
    cfg = synth.mlp(seed=1, sizes=(320, 192, 100, 10)) if workload == "mlp" else synth.fc_head(seed=0)
    layers = mlp_layers(3)
    in_dim = cfg["X"].shape[0]
    net = SparseNet(layers, cfg["W"], cfg["b"], cfg["X"].shape[1], (in_dim,), precision=1)
    assert net.fused
    net.x_in.copy_(torch.from_numpy(cfg["X"]))
    net.labels.copy_(torch.from_numpy(cfg["labels"]))
    onet = _oracle_net(layers, net)
    loss = net.step("prox", cfg["eta"], cfg["lambda"])
    torch.cuda.synchronize()
    assert net.ws.status()[0] == 0
    logits, _ = O.net_forward(onet, cfg["X"], cfg["X"].shape[1])
    oloss, _ = O.softmax_xent(logits, cfg["labels"])
    assert abs(float(loss[0].item()) - oloss) <= 2e-5 * max(1.0, abs(oloss))
    for pi, L in enumerate(net.params):
        W = onet.params[[i for i, l in enumerate(layers) if l["kind"] == "fc"][pi]]["W"]
        d = L["dpre"].cpu().numpy().reshape(W.rows, -1).astype(np.float64)
        x = L["xmat"].cpu().numpy().reshape(W.cols, -1).astype(np.float64)
        _assert_prox_within_bound(net.weights(pi), W, d, x, cfg["eta"], cfg["lambda"], f"layer {pi}")


@pytest.mark.parametrize("optimizer", ["adam", "rmsprop"])
def test_mlp_adaptive_prox_steps(C, optimizer):
    """The prox phase with Prox-ADAM (Algorithm 2) or Prox-RMSProp
    (Algorithm 1): three steps; each layer's G against the oracle on the GPU's
    own dL/dpre and input, and the update (CSR and moments) bit for bit against
    the oracle's adaptive step fed the GPU's G and the oracle's moments."""
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, mlp_layers
    cfg = synth.mlp(seed=2)
    layers = mlp_layers(3)
    net = SparseNet(layers, cfg["W"], cfg["b"], 256, (784,), precision=1, grad_per_layer=True,
                    optimizer=optimizer, beta1=0.9, beta2=0.999, rms_beta=0.9, eps=1e-8)
    net.x_in.copy_(torch.from_numpy(cfg["X"]))
    net.labels.copy_(torch.from_numpy(cfg["labels"]))
    moments = [{"m": np.zeros((L["W"][0].rows, L["W"][0].cols), F32),
                "v": np.zeros((L["W"][0].rows, L["W"][0].cols), F32)} for L in net.params]
    eta, lam = 1e-3, 0.05
    for t in range(1, 4):
        old = [_host_csr(net.weights(pi))[0] for pi in range(len(net.params))]
        net.step("prox", eta, lam)
        torch.cuda.synchronize()
        assert net.ws.status()[0] == 0 and net.t == t
        for pi, L in enumerate(net.params):
            G = L["G"].cpu().numpy()
            st = moments[pi]
            if optimizer == "adam":
                ref, st["m"], st["v"] = O.prox_adam_update_compact(old[pi], G, st["m"], st["v"], t, eta, lam, 0.9,
                                                                   0.999, 1e-8)
                np.testing.assert_array_equal(L["m"].cpu().numpy().view(np.uint32), st["m"].view(np.uint32))
            else:
                ref, st["v"] = O.prox_rmsprop_update_compact(old[pi], G, st["v"], eta, lam, 0.9, 1e-8)
            np.testing.assert_array_equal(L["v"].cpu().numpy().view(np.uint32), st["v"].view(np.uint32))
            _assert_csr_bits(net.weights(pi), ref)


@pytest.mark.parametrize("workload,fused,optimizer", [("mlp", True, "sgd"), ("mlp", False, "sgd"),
                                                      ("mlp", False, "adam"), ("fc_head", True, "sgd")])
def test_overlapped_backward_matches_one_stream(C, workload, fused, optimizer):
    """The prox phase with each layer's bias and weight update on a second
    stream (overlap) gives the same bits as the one-stream step: weights,
    transposed copies, biases and losses over two prox steps and a debias step."""
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, mlp_layers
    cfg = synth.mlp(seed=3) if workload == "mlp" else synth.fc_head(seed=0)
    in_dim, batch = cfg["X"].shape
    nets = []
    for ov in (False, True):
        net = SparseNet(mlp_layers(3), cfg["W"], cfg["b"], batch, (in_dim,), precision=1, fused=fused,
                        optimizer=optimizer, overlap=ov)
        net.x_in.copy_(torch.from_numpy(cfg["X"]))
        net.labels.copy_(torch.from_numpy(cfg["labels"]))
        nets.append(net)
    eta, lam = (1e-3, 0.05) if optimizer == "adam" else (cfg["eta"], cfg["lambda"])
    for phase in ("prox", "prox", "debias"):
        losses = [float(net.step(phase, eta, lam)[0].item()) for net in nets]
        torch.cuda.synchronize()
        assert losses[0] == losses[1]
        for net in nets:
            assert net.status()[0] == 0
        for pi in range(3):
            (a, ta), (b, tb) = nets[0].weights(pi).to_host(), nets[1].weights(pi).to_host()
            for x, y in zip(a, b):
                np.testing.assert_array_equal(x.view(np.uint32), y.view(np.uint32))
            if ta is not None:
                for x, y in zip(ta, tb):
                    np.testing.assert_array_equal(x.view(np.uint32), y.view(np.uint32))
            np.testing.assert_array_equal(nets[0].params[pi]["b"].cpu().numpy().view(np.uint32),
                                          nets[1].params[pi]["b"].cpu().numpy().view(np.uint32))
