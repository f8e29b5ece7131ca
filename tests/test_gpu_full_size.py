"""Oracle parity at full size: the 4096 x 4096 sweep layer and the
classifier-head step the bench times.

The sweep layer is drawn exactly as the sweep draws it (seed 0: weights at
density 1, 5, 20 or 50 % with uniform or Zipf(1.2) row lengths, then X and
dY of 1024 columns, then G, all N(0, 1); the products take the first n
columns), so these are the inputs behind the sweep's timings, run through the
same entry points and therefore the same kernel choices (unit counts, ring
chunks, vector and group widths, dense or sparse prox tiles).

The oracle is separable over output rows, so for the products it runs on a
fixed sample of 256 output rows (the 32 longest included: the Zipf head rows
that several work units share) rather than on all 4096; each sampled output
is compared element by element with the summation bound. The prox step is
compared bit for bit on the whole matrix, with and without the transposed
copy, at the workload's lambda = 1e-4 (the output is nearly dense) and at the
density-preserving lambda* (the (1 - d) quantile of |w - eta*G| / eta).
"""

import numpy as np
import pytest

import oracle as O
from tests.parity import TF32_OPERAND, U32, assert_close, csr_dense, gamma

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu
F32 = np.float32

SIDE = 4096
DENSITIES = (0.01, 0.05, 0.20, 0.50)
BATCHES = (1, 32, 256, 1024)


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import csrtrain
    csrtrain.lib()
    return csrtrain


_LAYER = {}


def _layer(density, zipf):
    """The sweep's inputs for one (density, row-length) case, in its draw order."""
    key = (density, zipf)
    if key not in _LAYER:
        from paper_1905_07931_gb300 import synth
        _LAYER.clear()
        rng = synth.rng_for(0)
        w = synth.masked_weights(rng, SIDE, SIDE, density, zipf=zipf)
        x = synth.std_normal(rng, SIDE, max(BATCHES))
        dy = synth.std_normal(rng, SIDE, max(BATCHES))
        g = synth.std_normal(rng, SIDE, SIDE)
        _LAYER[key] = (w, x, dy, g, synth.ETA, synth.LAMBDA)
    return _LAYER[key]


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _sample(lengths, count=256, longest=32, seed=12345):
    """A fixed sample of output rows: the `longest` rows by length, the first
    and last row, and random others, sorted."""
    rng = np.random.default_rng(seed)
    top = np.argsort(-np.asarray(lengths), kind="stable")[:longest]
    picks = set(int(i) for i in top) | {0, len(lengths) - 1}
    for i in rng.permutation(len(lengths)):
        if len(picks) >= count:
            break
        picks.add(int(i))
    return np.array(sorted(picks), dtype=np.int64)


def _rows_of(ref: "O.CSR", rows):
    """The CSR of the selected rows (same columns), and the positions of
    their entries in ref's arrays."""
    rp = ref.row_ptr.astype(np.int64)
    idx = np.concatenate([np.arange(rp[r], rp[r + 1]) for r in rows])
    lens = rp[rows + 1] - rp[rows]
    new_rp = np.zeros(len(rows) + 1, np.int64)
    new_rp[1:] = np.cumsum(lens)
    return O.CSR(len(rows), ref.cols, new_rp.astype(np.int32), ref.col_idx[idx], ref.val[idx]), idx


def _lambda_star(w, g, eta, density):
    """Density-preserving lambda: the (1 - d) quantile of |w - eta*G| / eta."""
    z = np.abs(w.astype(np.float64) - eta * g.astype(np.float64)) / eta
    return float(np.quantile(z, 1.0 - density))


@pytest.mark.parametrize("zipf", [False, True], ids=["uniform", "zipf"])
@pytest.mark.parametrize("density", DENSITIES)
def test_products_on_the_sweep_layer(C, density, zipf):
    """spmm_fwd, spmm_bwd_t and weight_grad_sddmm at n = 1, 32, 256, 1024
    (Sections 3.2.1, 3.2.2 and 2.4) on sampled output rows."""
    w, x_all, dy_all, _, _, _ = _layer(density, zipf)
    ref = O.csr_from_dense(w)
    ws = C.Workspace(SIDE, SIDE, max(BATCHES))
    W = C.CSR(SIDE, SIDE, capacity=max(ref.nnz, 1))
    C.csr_from_dense(_dev(w), W, ws)
    assert W.nnz() == ref.nnz
    lens = np.diff(ref.row_ptr.astype(np.int64))
    clens = np.bincount(ref.col_idx, minlength=SIDE)
    rows = _sample(lens)
    cols = _sample(clens)
    sub_r, idx_r = _rows_of(ref, rows)
    sub_c = O.csr_from_dense(w[:, cols])        # W restricted to the sampled columns
    rows_d, cols_d, idx_d = _dev(rows), _dev(cols), _dev(idx_r)
    for n in BATCHES:
        x = np.ascontiguousarray(x_all[:, :n])
        dy = np.ascontiguousarray(dy_all[:, :n])
        xd, dyd = _dev(x), _dev(dy)
        y = torch.empty(SIDE, n, device="cuda")
        C.spmm_fwd(W, xd, y, ws)
        assert_close(y[rows_d].cpu().numpy(), O.spmm_fwd(sub_r, x),
                     lambda: O.spmm_fwd(O.csr_abs(sub_r), np.abs(x)), lens[rows][:, None],
                     what=f"spmm_fwd n={n}")
        dx = torch.empty(SIDE, n, device="cuda")
        C.spmm_bwd_t(W, dyd, dx, ws)
        assert_close(dx[cols_d].cpu().numpy(), O.spmm_bwd_t(sub_c, dy),
                     lambda: O.spmm_bwd_t(O.csr_abs(sub_c), np.abs(dy)), clens[cols][:, None],
                     what=f"spmm_bwd_t n={n}")
        g = torch.empty(max(ref.nnz, 1), device="cuda")
        C.weight_grad_sddmm(W, dyd, xd, g, ws)
        dy_r = dy[rows]
        assert_close(g[idx_d].cpu().numpy(), O.weight_grad_sddmm(sub_r, dy_r, x),
                     lambda: O.weight_grad_sddmm(sub_r, np.abs(dy_r), np.abs(x)), n,
                     what=f"sddmm n={n}")
        assert ws.status()[0] == 0


def _assert_same_csr(out, ref, t_ref, transposed):
    (rp, ci, v), t = out.to_host()
    np.testing.assert_array_equal(rp, ref.row_ptr)
    np.testing.assert_array_equal(ci, ref.col_idx)
    np.testing.assert_array_equal(v.view(np.uint32), ref.val.astype(F32).view(np.uint32))
    if transposed:
        for got, want in zip(t, t_ref):
            np.testing.assert_array_equal(got.view(np.uint32), np.asarray(want).astype(got.dtype).view(np.uint32))


@pytest.mark.parametrize("zipf", [False, True], ids=["uniform", "zipf"])
@pytest.mark.parametrize("density", DENSITIES)
def test_prox_on_the_sweep_layer(C, density, zipf):
    """prox_update_compact (Section 2.2, Eq. prox, Section 3.3) on the whole
    layer, bit for bit, at lambda = 1e-4 and at lambda*, each with and without
    the transposed copy."""
    w, _, _, g, eta, lam = _layer(density, zipf)
    ref_in = O.csr_from_dense(w)
    ws = C.Workspace(SIDE, SIDE, 1)
    W = C.CSR(SIDE, SIDE, capacity=max(ref_in.nnz, 1), transposed=False)
    C.csr_from_dense(_dev(w), W, ws)
    gd = _dev(g)
    for lam_v in (lam, _lambda_star(w, g, eta, density)):
        ref = O.prox_update_compact(ref_in, g, eta, lam_v)
        t_ref = O.csr_transpose(ref)
        if lam_v != lam:
            assert abs(ref.nnz - density * SIDE * SIDE) <= 0.01 * density * SIDE * SIDE + 2
        for transposed in (True, False):
            out = C.CSR(SIDE, SIDE, transposed=transposed)
            C.prox_update_compact(W, gd, eta, lam_v, out, ws)
            assert ws.status()[0] == 0
            _assert_same_csr(out, ref, t_ref, transposed)
            del out
            torch.cuda.empty_cache()


def test_prox_beyond_the_place_kernels_prefix(C):
    """prox_update_compact on a layer of 4100 x 8192 (one row per tile, 4100
    tiles: more than the place kernel sums counts over itself, so the row
    pointers come from a scan of the row counts), bit for bit at lambda =
    1e-4 and at lambda*, with and without the transposed copy."""
    from paper_1905_07931_gb300 import synth
    m, k, density = 4100, 8192, 0.05
    rng = synth.rng_for(7)
    w = synth.masked_weights(rng, m, k, density, zipf=False)
    g = synth.std_normal(rng, m, k)
    eta, lam = synth.ETA, synth.LAMBDA
    ref_in = O.csr_from_dense(w)
    ws = C.Workspace(m, k, 1)
    W = C.CSR(m, k, capacity=max(ref_in.nnz, 1), transposed=False)
    C.csr_from_dense(_dev(w), W, ws)
    gd = _dev(g)
    for lam_v in (lam, _lambda_star(w, g, eta, density)):
        ref = O.prox_update_compact(ref_in, g, eta, lam_v)
        t_ref = O.csr_transpose(ref)
        for transposed in (True, False):
            out = C.CSR(m, k, transposed=transposed)
            C.prox_update_compact(W, gd, eta, lam_v, out, ws)
            assert ws.status()[0] == 0
            _assert_same_csr(out, ref, t_ref, transposed)
            del out
            torch.cuda.empty_cache()


# ---------------------------------------------------------------------------
# The classifier-head step (9216-4096-4096-1000, batch 256): the fused
# gradient + prox op against the unfused calls at the bench's own shapes
# ---------------------------------------------------------------------------

def _columns_strictly_ascending(row_ptr, col_idx):
    rp = row_ptr.astype(np.int64)
    if len(col_idx) < 2:
        return True
    d = np.diff(col_idx.astype(np.int64))
    starts = np.zeros(len(col_idx), dtype=bool)
    starts[rp[1:-1][rp[1:-1] < len(col_idx)]] = True
    return bool(np.all((d > 0) | starts[1:]))


def _prox_band(w_gpu_host, W_old, d, x, eta, lam):
    """The fused prox step against the oracle's float64 G of the same dL/dpre
    and layer input (G is never written, so it cannot be re-fed): every entry
    whose |w - eta*G| lies farther from eta*lambda than the TF32 error band dz
    takes the oracle's keep decision, every kept value lies within dz of the
    soft threshold. Returns (entries kept, entries inside the band)."""
    rp, ci, v = w_gpu_host
    M, K = W_old.rows, W_old.cols
    n = x.shape[1]
    G = O.weight_grad_dense(d, x)
    S = O.weight_grad_dense(np.abs(d), np.abs(x))
    tol = gamma(n + 1) * S + U32 * np.abs(G) + 2 * TF32_OPERAND * S + 1e-30
    w0 = csr_dense(W_old.row_ptr, W_old.col_idx, W_old.val, M, K).astype(np.float64)
    thr = float(np.float32(eta) * np.float32(lam))
    z = w0 - eta * G
    dz = 2.0 * (eta * tol + U32 * (eta * np.abs(G) + np.abs(z))) + 1e-30
    keep = np.zeros((M, K), dtype=bool)
    keep[np.repeat(np.arange(M), np.diff(rp.astype(np.int64))), ci] = True
    band = np.abs(np.abs(z) - thr) <= dz
    wrong = ~band & (keep != (np.abs(z) > thr))
    assert not wrong.any(), f"{int(wrong.sum())} keep decisions outside the TF32 band"
    vg = csr_dense(rp, ci, v, M, K).astype(np.float64)
    want = z - np.sign(z) * thr
    assert np.all(np.abs(vg - want)[keep] <= dz[keep] + U32 * np.abs(want[keep])), "kept values beyond the band"
    return int(keep.sum()), int(band.sum())


def test_fused_gradient_prox_at_the_bench_step(C, record_property):
    """One prox step of the classifier head as the bench runs it (fused
    weight_grad_prox_update on every layer, TF32): each layer's output CSR,
    and its transposed copy where the step keeps one, is bit-identical to
    weight_grad_dense (TF32) + prox_update_compact fed the same dL/dpre and
    layer input; against the oracle's float64 gradient, keep decisions
    outside the TF32 band are exact and the entries inside the band are
    counted (reported as a test property and printed: about 2% of the
    4096 x 9216 layer's entries, since truncating both operands to TF32
    widens the band to about 2^-9 of sum |dY X| around the threshold; the
    test only checks that it stays below 10%)."""
    from paper_1905_07931_gb300 import synth
    from paper_1905_07931_gb300.train import SparseNet, mlp_layers
    cfg = synth.fc_head(seed=0)
    net = SparseNet(mlp_layers(3), cfg["W"], cfg["b"], 256, (9216,), precision=C.CSRT_PREC_TF32)
    assert net.fused
    net.x_in.copy_(torch.from_numpy(cfg["X"]))
    net.labels.copy_(torch.from_numpy(cfg["labels"]))
    eta, lam = cfg["eta"], cfg["lambda"]
    net.step("prox", eta, lam)
    torch.cuda.synchronize()
    assert net.ws.status()[0] == 0
    for li, L in enumerate(net.params):
        W_in, W_fused = L["W"][1 - L["cur"]], L["W"][L["cur"]]
        M, K = W_in.rows, W_in.cols
        G = torch.empty(M, K, device="cuda")
        C.weight_grad_dense(L["dpre"], L["xmat"], G, net.ws, precision=C.CSRT_PREC_TF32)
        unf = C.CSR(M, K, transposed=W_fused.transposed)
        C.prox_update_compact(W_in, G, eta, lam, unf, net.ws)
        assert net.ws.status()[0] == 0
        (rp, ci, v), t = W_fused.to_host()
        (rp2, ci2, v2), t2 = unf.to_host()
        np.testing.assert_array_equal(rp, rp2)
        np.testing.assert_array_equal(ci, ci2)
        np.testing.assert_array_equal(v.view(np.uint32), v2.view(np.uint32))
        if W_fused.transposed:
            for a, b in zip(t, t2):
                np.testing.assert_array_equal(a.view(np.uint32), b.view(np.uint32))
        assert rp[0] == 0 and np.all(np.diff(rp.astype(np.int64)) >= 0)
        assert _columns_strictly_ascending(rp, ci)
        (orp, oci, ov), _ = W_in.to_host()
        old = O.CSR(M, K, orp.copy(), oci.copy(), ov.copy())
        d = L["dpre"].cpu().numpy().reshape(M, -1).astype(np.float64)
        x = L["xmat"].cpu().numpy().reshape(K, -1).astype(np.float64)
        kept, in_band = _prox_band((rp, ci, v), old, d, x, eta, lam)
        record_property(f"layer{li}_kept", kept)
        record_property(f"layer{li}_in_band", in_band)
        print(f"layer {li} ({M}x{K}): {kept} kept, {in_band} of {M * K} entries inside the TF32 band")
        assert in_band <= 0.1 * M * K
        del G, unf
