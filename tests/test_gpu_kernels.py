"""Parity of every C-ABI call against the CPU oracle, on seeded inputs.

Sizes span several compaction tiles (4096 entries) and SpMM units with a
ragged tail, empty rows, power-law rows, odd column counts and the degenerate
cases (empty matrix, all-zero, fully dense, n = 1). Integer arrays are
compared bit for bit; the prox step is bit-exact when fed the same G.
"""

import json
import os

import numpy as np
import pytest

import oracle as O
from tests.parity import assert_close, csr_dense

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GOLD = os.path.join(os.path.dirname(__file__), "golden")
F32 = np.float32


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import csrtrain
    csrtrain.lib()
    return csrtrain


def _ws(C, rows, cols, n):
    return C.Workspace(max(rows, 1), max(cols, 1), max(n, 1))


def _sparse(rng, m, k, density, zipf=False):
    from paper_1905_07931_gb300 import synth
    return synth.masked_weights(rng, m, k, density, std=1.0, zipf=zipf)


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _gpu_csr(C, dense, ws, transposed=True, capacity=None):
    m, k = dense.shape
    w = C.CSR(m, k, capacity=capacity, transposed=transposed)
    C.csr_from_dense(_dev(dense.astype(F32)), w, ws)
    return w


def _check_csr_equal(w, ref: "O.CSR", transposed=True):
    (rp, ci, v), t = w.to_host()
    np.testing.assert_array_equal(rp, ref.row_ptr)
    np.testing.assert_array_equal(ci, ref.col_idx)
    np.testing.assert_array_equal(v.view(np.uint32), ref.val.astype(F32).view(np.uint32))
    if transposed:
        trp, tci, tv, tpos = O.csr_transpose(ref)
        np.testing.assert_array_equal(t[0], trp)
        np.testing.assert_array_equal(t[1], tci)
        np.testing.assert_array_equal(t[2].view(np.uint32), tv.astype(F32).view(np.uint32))
        np.testing.assert_array_equal(t[3], tpos)


# --- csr_from_dense / csr_transpose -----------------------------------------

def test_worked_example_on_gpu(C):
    with open(os.path.join(GOLD, "csr_worked_example.json")) as f:
        d = json.load(f)
    a = np.array(d["dense"], dtype=F32)
    ws = _ws(C, 4, 4, 1)
    w = _gpu_csr(C, a, ws)
    (rp, ci, v), t = w.to_host()
    assert rp.tolist() == d["row_ptrs"]
    assert ci.tolist() == d["col_indices"]
    assert v.tolist() == d["elements"]
    h = d["hand_derived"]
    assert t[0].tolist() == h["transpose_row_ptrs"]
    assert t[1].tolist() == h["transpose_col_indices"]
    assert t[2].tolist() == h["transpose_elements"]
    assert t[3].tolist() == h["transpose_pos_of_each_csr_entry"]
    y = torch.zeros(4, 1, device="cuda")
    C.spmm_fwd(w, torch.ones(4, 1, device="cuda"), y, ws)
    assert y[:, 0].cpu().tolist() == h["A_times_ones"]
    C.spmm_bwd_t(w, torch.ones(4, 1, device="cuda"), y, ws)
    assert y[:, 0].cpu().tolist() == h["At_times_ones"]


@pytest.mark.parametrize("m,k,density", [(1, 1, 1.0), (3, 5, 0.5), (33, 129, 0.3), (300, 784, 0.1),
                                         (17, 1, 0.5), (5, 3, 1.0), (41, 9216, 0.05), (64, 64, 0.0),
                                         (2, 70000, 0.01), (257, 31, 0.9)])
def test_csr_from_dense_bit_exact(C, m, k, density):
    rng = np.random.default_rng(m * 7 + k)
    a = _sparse(rng, m, k, density)
    if m > 2:
        a[1, :] = 0.0
        a[m - 1, :] = 0.0
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    _check_csr_equal(w, O.csr_from_dense(a))
    assert ws.status()[0] == 0


def test_csr_from_dense_signed_zero_nan_inf(C):
    a = np.array([[-0.0, 1.0, np.nan, 0.0, np.inf, -np.inf, -2.0]], dtype=F32)
    ws = _ws(C, 1, 7, 1)
    w = _gpu_csr(C, a, ws, transposed=False)
    (rp, ci, v), _ = w.to_host()
    assert ci.tolist() == [1, 2, 4, 5, 6]
    assert rp.tolist() == [0, 5]


def test_csr_capacity_overflow_is_reported_and_clamped(C):
    rng = np.random.default_rng(3)
    a = _sparse(rng, 40, 300, 0.5)
    nnz = int((a != 0).sum())
    ws = _ws(C, 40, 300, 1)
    w = _gpu_csr(C, a, ws, transposed=False, capacity=nnz // 2)
    flags, required = ws.status()
    assert flags & C.CSRT_DEV_CAPACITY
    assert required == nnz
    rp = w.row_ptr.cpu().numpy()
    assert (np.diff(rp) >= 0).all() and rp[-1] == nnz // 2
    ref = O.csr_from_dense(a)
    np.testing.assert_array_equal(w.col_idx.cpu().numpy()[: nnz // 2], ref.col_idx[: nnz // 2])
    ws.clear_status()
    assert ws.status()[0] == 0


def test_empty_matrix_shapes(C):
    ws = _ws(C, 8, 8, 4)
    w = C.CSR(0, 5, transposed=True)
    C.csr_from_dense(torch.zeros(1, device="cuda"), w, ws)
    assert w.row_ptr.cpu().tolist() == [0]
    assert w.t_row_ptr.cpu().tolist() == [0] * 6
    w2 = C.CSR(4, 0, transposed=False)
    C.csr_from_dense(torch.zeros(1, device="cuda"), w2, ws)
    assert w2.row_ptr.cpu().tolist() == [0] * 5


# --- spmm_fwd / spmm_bwd_t ----------------------------------------------------

SPMM_CASES = [
    (300, 784, 64, 0.1, False),
    (37, 53, 1, 0.3, False),
    (37, 53, 3, 0.3, False),
    (129, 257, 32, 0.2, False),
    (129, 257, 70, 0.2, False),
    (500, 300, 256, 0.05, True),
    (64, 2000, 130, 0.5, True),
    (20, 25, 4100, 0.3, False),
    (4, 9, 1, 1.0, False),
    (50, 40, 7, 0.0, False),
    (1000, 600, 1024, 0.02, True),
    # long rows cut by many work units, one float4 per lane, a ragged
    # second n-tile, and a larger uniform case
    (300, 5000, 256, 0.1, False),
    (129, 1000, 128, 0.2, False),
    (257, 300, 384, 0.3, True),
    (2048, 1024, 256, 0.05, False),
    # tall products: thousands of rows, power-law rows at n = 128, and a
    # transposed product with 9000 output rows
    (4100, 700, 256, 0.05, False),
    (7400, 257, 128, 0.2, True),
    (300, 9000, 256, 0.05, False),
    # narrow products (G lanes per nonzero, G*VW >= n): every group width and
    # vector width, rows of thousands of entries cut by many units, power-law
    # rows, empty rows, and tails shorter than one batch
    (64, 20000, 1, 0.5, False),
    (2000, 3000, 1, 0.05, True),
    (1500, 1100, 2, 0.2, False),
    (700, 900, 3, 0.1, True),
    (300, 5000, 4, 0.3, False),
    (257, 700, 5, 0.2, False),
    (400, 2500, 8, 0.4, True),
    (129, 257, 12, 0.2, False),
    (600, 4000, 16, 0.1, False),
    (300, 800, 24, 0.3, True),
    (129, 4000, 32, 0.5, False),
    (1000, 600, 48, 0.1, True),
    (300, 2000, 64, 0.2, False),
    (90, 70, 9, 0.0, False),
    # wide products with thousands of rows at n = 128 to 1024: power-law
    # rows, a ragged last block of X rows, densities from 2% to 30%
    (2600, 300, 256, 0.2, True),
    (5000, 600, 128, 0.3, True),
    (2500, 2000, 256, 0.04, False),
    (2500, 500, 256, 0.02, False),
    (2432, 130, 1024, 0.3, False),
]


@pytest.mark.parametrize("m,k,n,density,zipf", SPMM_CASES)
def test_spmm_fwd_and_bwd_against_oracle(C, m, k, n, density, zipf):
    rng = np.random.default_rng(m + 3 * k + 7 * n)
    a = _sparse(rng, m, k, density, zipf)
    if m > 4:
        a[2, :] = 0.0
    x = rng.standard_normal((k, n)).astype(F32)
    dy = rng.standard_normal((m, n)).astype(F32)
    ws = _ws(C, m, k, n)
    w = _gpu_csr(C, a, ws)
    ref = O.csr_from_dense(a)
    y = torch.zeros(m, n, device="cuda")
    C.spmm_fwd(w, _dev(x), y, ws)
    lens = np.diff(ref.row_ptr)[:, None]
    assert_close(y.cpu().numpy(), O.spmm_fwd(ref, x), O.spmm_fwd(O.csr_abs(ref), np.abs(x)), lens,
                 what="spmm_fwd")
    dx = torch.zeros(k, n, device="cuda")
    C.spmm_bwd_t(w, _dev(dy), dx, ws)
    clens = np.bincount(ref.col_idx, minlength=k)[:, None]
    assert_close(dx.cpu().numpy(), O.spmm_bwd_t(ref, dy), O.spmm_bwd_t(O.csr_abs(ref), np.abs(dy)), clens,
                 what="spmm_bwd_t")
    assert ws.status()[0] == 0


class _Shifted:
    """A CSR whose index and value arrays start 4 bytes past a 16-byte
    boundary (a caller's sub-array): the narrow kernel's bulk copies need
    16-byte alignment, so the library takes the 32-lane kernel for it."""

    def __init__(self, C, w):
        nnz = w.nnz()
        self.rows, self.cols = w.rows, w.cols
        self._c = torch.zeros(nnz + 1, dtype=torch.int32, device="cuda")
        self._v = torch.zeros(nnz + 1, dtype=torch.float32, device="cuda")
        self._c[1:].copy_(w.col_idx[:nnz])
        self._v[1:].copy_(w.val[:nnz])
        assert (self._c[1:].data_ptr() % 16) == 4 and (self._v[1:].data_ptr() % 16) == 4
        self._s = C.csrt_csr(w.rows, w.cols, max(nnz, 1), C._ptr(w.row_ptr), C._ptr(self._c[1:]),
                             C._ptr(self._v[1:]), None, None, None, None)
        self._keep = w

    @property
    def struct(self):
        import ctypes
        return ctypes.byref(self._s)


@pytest.mark.parametrize("n", [1, 3, 8, 16])
def test_spmm_narrow_unaligned_csr_arrays(C, n):
    m, k = 600, 700
    rng = np.random.default_rng(90 + n)
    a = _sparse(rng, m, k, 0.2)
    x = rng.standard_normal((k, n)).astype(F32)
    ws = _ws(C, m, k, n)
    w = _gpu_csr(C, a, ws)
    ref = O.csr_from_dense(a)
    want = torch.zeros(m, n, device="cuda")
    C.spmm_fwd(w, _dev(x), want, ws)            # aligned arrays: the narrow kernel
    got = torch.zeros(m, n, device="cuda")
    C.spmm_fwd(_Shifted(C, w), _dev(x), got, ws)   # shifted arrays: the 32-lane kernel
    lens = np.diff(ref.row_ptr)[:, None]
    for y in (want, got):
        assert_close(y.cpu().numpy(), O.spmm_fwd(ref, x), O.spmm_fwd(O.csr_abs(ref), np.abs(x)), lens,
                     what="spmm_fwd")
    assert ws.status()[0] == 0


@pytest.mark.parametrize("m,k,n,zipf", [(700, 900, 256, True), (129, 257, 70, False), (50, 40, 1, False),
                                         (300, 784, 64, False), (4100, 4100, 256, False), (5000, 5000, 128, True)])
def test_fused_epilogues_match_unfused(C, m, k, n, zipf):
    rng = np.random.default_rng(m + k + n)
    a = _sparse(rng, m, k, 0.1, zipf)
    x = _dev(rng.standard_normal((k, n)).astype(F32))
    dy = _dev(rng.standard_normal((m, n)).astype(F32))
    bias = _dev(rng.standard_normal(m).astype(F32))
    below = _dev(np.maximum(rng.standard_normal((k, n)), 0).astype(F32))
    ws = _ws(C, m, k, n)
    w = _gpu_csr(C, a, ws)
    for relu in (False, True):
        y_ref = torch.zeros(m, n, device="cuda")
        C.spmm_fwd(w, x, y_ref, ws)
        C.bias_act_fwd(y_ref, bias, relu)
        y = torch.zeros(m, n, device="cuda")
        C.spmm_fwd_bias_act(w, x, bias, relu, y, ws)
        np.testing.assert_array_equal(y.cpu().numpy().view(np.uint32), y_ref.cpu().numpy().view(np.uint32))
    dx_ref = torch.zeros(k, n, device="cuda")
    C.spmm_bwd_t(w, dy, dx_ref, ws)
    C.relu_bwd(dx_ref, below)
    dx = torch.zeros(k, n, device="cuda")
    C.spmm_bwd_t_relu(w, dy, below, dx, ws)
    np.testing.assert_array_equal(dx.cpu().numpy().view(np.uint32), dx_ref.cpu().numpy().view(np.uint32))


@pytest.mark.parametrize("m,k,n", [(700, 900, 1), (700, 900, 8), (700, 900, 32), (700, 900, 96), (700, 900, 256),
                                   (5000, 900, 256)])
def test_spmm_is_deterministic(C, m, k, n):
    rng = np.random.default_rng(11)
    a = _sparse(rng, m, k, 0.08, zipf=True)
    x = _dev(rng.standard_normal((k, n)).astype(F32))
    ws = _ws(C, m, k, n)
    w = _gpu_csr(C, a, ws)
    ys = []
    for _ in range(3):
        y = torch.zeros(m, n, device="cuda")
        C.spmm_fwd(w, x, y, ws)
        ys.append(y.cpu().numpy())
    np.testing.assert_array_equal(ys[0].view(np.uint32), ys[1].view(np.uint32))
    np.testing.assert_array_equal(ys[0].view(np.uint32), ys[2].view(np.uint32))


# --- weight gradients ----------------------------------------------------------

@pytest.mark.parametrize("m,k,n", [(300, 784, 64), (10, 500, 128), (20, 25, 9000), (129, 67, 33),
                                   (1, 1, 1), (256, 512, 256)])
@pytest.mark.parametrize("prec", [0, 1])
def test_weight_grad_dense(C, m, k, n, prec):
    rng = np.random.default_rng(m + k + n + prec)
    dy = rng.standard_normal((m, n)).astype(F32)
    x = rng.standard_normal((k, n)).astype(F32)
    ws = _ws(C, m, k, n)
    g = torch.zeros(m, k, device="cuda")
    C.weight_grad_dense(_dev(dy), _dev(x), g, ws, precision=prec)
    ref = O.weight_grad_dense(dy, x)
    bound = O.weight_grad_dense(np.abs(dy), np.abs(x))
    assert_close(g.cpu().numpy(), ref, bound, n, rtol=1e-3 if prec else 1e-4, tf32=bool(prec),
                 what=f"weight_grad_dense prec={prec}")


@pytest.mark.parametrize("m,k,n,density,zipf", [(300, 784, 64, 0.1, False), (100, 300, 256, 0.09, True),
                                                (20, 25, 9000, 0.3, False), (50, 40, 1, 0.5, False),
                                                (33, 17, 5, 0.0, False),
                                                # every group width, float4 / float2 / scalar rows of X,
                                                # long and power-law rows, n walked in several tiles
                                                (64, 20000, 1, 0.5, False), (2000, 3000, 1, 0.05, True),
                                                (700, 900, 2, 0.1, True), (300, 5000, 3, 0.2, False),
                                                (400, 2500, 8, 0.3, True), (129, 4000, 32, 0.5, False),
                                                (300, 900, 33, 0.2, False), (257, 700, 64, 0.2, True),
                                                (300, 800, 130, 0.1, False), (500, 3000, 256, 0.05, True),
                                                (100, 300, 1024, 0.2, False), (60, 90, 1030, 0.3, True)])
def test_weight_grad_sddmm(C, m, k, n, density, zipf):
    rng = np.random.default_rng(m * k + n)
    a = _sparse(rng, m, k, density, zipf)
    dy = rng.standard_normal((m, n)).astype(F32)
    x = rng.standard_normal((k, n)).astype(F32)
    ws = _ws(C, m, k, n)
    w = _gpu_csr(C, a, ws, transposed=False)
    ref = O.csr_from_dense(a)
    g = torch.zeros(max(ref.nnz, 1), device="cuda")
    C.weight_grad_sddmm(w, _dev(dy), _dev(x), g, ws)
    got = g.cpu().numpy()[: ref.nnz]
    assert_close(got, O.weight_grad_sddmm(ref, dy, x), O.weight_grad_sddmm(ref, np.abs(dy), np.abs(x)), n,
                 what="sddmm")
    # the same values as the dense gradient read at the pattern
    dense = O.weight_grad_dense(dy, x)
    assert_close(got, dense[ref.row_of_each_entry(), ref.col_idx],
                 O.weight_grad_dense(np.abs(dy), np.abs(x))[ref.row_of_each_entry(), ref.col_idx], n,
                 what="sddmm vs masked dense")


# --- prox_update_compact / debias_update ---------------------------------------

def test_prox_hand_cases_on_gpu(C):
    with open(os.path.join(GOLD, "soft_threshold_cases.json")) as f:
        d = json.load(f)
    ws_ = np.array([[c["w"] for c in d["cases"]]], dtype=F32)
    gs = np.array([[c["g"] for c in d["cases"]]], dtype=F32)
    ws = _ws(C, 1, ws_.shape[1], 1)
    w = _gpu_csr(C, ws_, ws)
    out = C.CSR(1, ws_.shape[1])
    C.prox_update_compact(w, _dev(gs), d["eta"], d["lambda"], out, ws)
    (rp, ci, v), _ = out.to_host()
    dense = csr_dense(rp, ci, v, 1, ws_.shape[1])[0]
    for j, c in enumerate(d["cases"]):
        assert (dense[j] != 0) == c["kept"], c
        assert dense[j] == F32(c["out"]), c


@pytest.mark.parametrize("m,k,density,gscale,eta,lam", [
    (300, 784, 0.1, 1.0, 0.01, 1e-4),
    (300, 784, 0.1, 1e-3, 0.5, 1e-2),
    (37, 4099, 0.3, 0.1, 0.1, 0.3),
    (1, 5000, 0.5, 1.0, 0.01, 50.0),
    (4097, 3, 0.6, 1.0, 0.2, 0.5),
    (100, 300, 0.09, 1.0, 0.0, 1e-4),
    (64, 64, 0.0, 0.0, 0.1, 0.0),
    (500, 800, 0.08, 1e-2, 0.01, 1e-2),
    (1001, 784, 0.1, 1.0, 0.01, 1e-2),
    (333, 64, 0.4, 1.0, 0.1, 1.0),
    (3, 16384, 0.02, 1.0, 0.01, 0.5),
    (2, 16388, 0.02, 1.0, 0.01, 0.5),
    (2, 20000, 0.3, 1.0, 0.01, 0.5),
    (4100, 512, 0.05, 1.0, 0.01, 1e-4),
    (700, 900, 0.5, 0.1, 0.1, 1.0),
    (20000, 784, 0.05, 1.0, 0.01, 1e-2),   # 2000 row tiles: several per resident block
    (2000, 20, 0.3, 1.0, 0.01, 1e-4),      # dense tiles of short rows: a 32-entry step spans 2-3 rows
    (3000, 8, 0.5, 1.0, 0.01, 1e-4),       # ... 4-5 rows
    (1500, 36, 0.2, 1.0, 0.01, 1e-4),      # K >= 32, not a multiple of 32
    (1500, 9216, 0.05, 1.0, 0.01, 1e-4),   # one-row tiles, dense output
])
def test_prox_bit_exact(C, m, k, density, gscale, eta, lam):
    rng = np.random.default_rng(m + k)
    a = _sparse(rng, m, k, density)
    g = (rng.standard_normal((m, k)) * gscale).astype(F32)
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(m, k)
    C.prox_update_compact(w, _dev(g), eta, lam, out, ws)
    ref = O.prox_update_compact(O.csr_from_dense(a), g, eta, lam)
    _check_csr_equal(out, ref)
    assert ws.status()[0] == 0


def _largest_below(eta, thr):
    """The largest float32 x >= 0 with fl(eta*x) <= thr (None if none), by
    walking float32 bit patterns from fl(thr/eta): the decision boundary of
    |fl(eta*G)| > thr in G, found with numpy's float32 products."""
    eta, thr = np.float32(eta), np.float32(thr)
    ok = lambda u: np.float32(eta * np.array([u], np.uint32).view(np.float32)[0]) <= thr
    if not ok(0):
        return None
    u = int(min(np.array([thr / eta], np.float32).view(np.uint32)[0], 0x7F800000))
    while u > 0 and not ok(u):
        u -= 1
    while u < 0x7F800000 and ok(u + 1):
        u += 1
    return np.array([u], np.uint32).view(np.float32)[0]


@pytest.mark.parametrize("eta,lam", [(0.01, 1e-4), (0.013, 7.7e-5), (1e-3, 1e-38), (3.0, 1e-7), (0.01, 0.0)])
@pytest.mark.parametrize("m,k", [(64, 256), (3, 9216)])
def test_prox_keep_boundary(C, eta, lam, m, k):
    """Gradients on both sides of the keep boundary: off the pattern an entry
    is kept iff |fl(eta*G)| > fl(eta*lambda) (Section 2.2's soft threshold
    applied to 0 - eta*G). G takes the largest magnitude that is dropped, the
    next float up, their negatives and a few patterns around them, on stored
    and unstored positions; bit-exact against the oracle."""
    thr = np.float32(np.float32(eta) * np.float32(lam))
    b = _largest_below(eta, thr)
    assert b is not None and np.float32(np.float32(eta) * np.nextafter(b, np.float32(np.inf))) > thr
    near = np.array([b], np.float32).view(np.uint32)[0].astype(np.int64) + np.arange(-3, 4)
    near = near[(near >= 0) & (near < 0x7F800000)].astype(np.uint32).view(np.float32)
    rng = np.random.default_rng(int(eta * 1e4) + m)
    vals = np.concatenate([near, -near])
    g = rng.choice(vals, size=(m, k)).astype(F32)
    g[:, ::7] = (rng.standard_normal((m, (k + 6) // 7)) * 4 * max(b, 1e-30)).astype(F32)
    a = _sparse(rng, m, k, 0.1)
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(m, k)
    C.prox_update_compact(w, _dev(g), eta, lam, out, ws)
    ref = O.prox_update_compact(O.csr_from_dense(a), g, eta, lam)
    _check_csr_equal(out, ref)
    kept = int(ref.row_ptr[-1])
    assert 0 < kept < m * k   # both decisions occur
    assert ws.status()[0] == 0


@pytest.mark.parametrize("eta,lam", [(0.0, 1e-4), (0.01, 0.0), (1e-3, 1e-38), (0.5, 1e30), (1e20, 1e20),
                                     (3.0, 1e-7)])
def test_prox_threshold_edges(C, eta, lam):
    """prox_update_compact bit-exact with the oracle at eta = 0, lambda = 0, a
    subnormal threshold, a threshold above every product and an infinite one,
    with infinite and NaN gradients among the entries; NaN in w - eta*G is
    flagged (with eta = 0 an infinite gradient gives NaN too)."""
    m, k = 300, 512
    rng = np.random.default_rng(int(eta * 7) % 1000 + 3)
    a = _sparse(rng, m, k, 0.1)
    g = rng.standard_normal((m, k)).astype(F32)
    g[5, 7] = np.inf
    g[9, 100] = -np.inf
    g[11, 3] = np.nan
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(m, k)
    C.prox_update_compact(w, _dev(g), eta, lam, out, ws)
    with np.errstate(invalid="ignore", over="ignore"):   # inf - inf and 0 * inf in the oracle's float32 rules
        ref = O.prox_update_compact(O.csr_from_dense(a), g, eta, lam)
    _check_csr_equal(out, ref)
    assert ws.status()[0] & C.CSRT_DEV_NONFINITE
    ws.clear_status()
    g2 = np.where(np.isfinite(g), g, 0).astype(F32)
    g2[5, 7] = np.inf                     # an infinity alone: flagged only where eta * Inf is NaN
    out2 = C.CSR(m, k)
    C.prox_update_compact(w, _dev(g2), eta, lam, out2, ws)
    with np.errstate(invalid="ignore", over="ignore"):
        ref2 = O.prox_update_compact(O.csr_from_dense(a), g2, eta, lam)
    _check_csr_equal(out2, ref2)
    assert bool(ws.status()[0] & C.CSRT_DEV_NONFINITE) == (eta == 0.0)   # w - fl(0 * Inf) is NaN


@pytest.mark.parametrize("m,k,transposed", [(3000, 512, True), (800, 9216, False), (5000, 300, True)])
def test_prox_mixed_dense_and_sparse_tiles(C, m, k, transposed):
    """Rows whose G is large keep nearly every entry (their tiles take the
    one-entry-per-lane pass 2), rows whose G is tiny keep only some stored
    weights (four-entries-per-lane pass 2): both forms in one call, bit-exact."""
    rng = np.random.default_rng(m + k)
    a = _sparse(rng, m, k, 0.1)
    scale = np.where((np.arange(m) // 37) % 2 == 0, 1.0, 1e-4).astype(F32)[:, None]
    g = (rng.standard_normal((m, k)).astype(F32) * scale).astype(F32)
    eta, lam = 0.01, 1e-2
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(m, k, transposed=transposed)
    C.prox_update_compact(w, _dev(g), eta, lam, out, ws)
    ref = O.prox_update_compact(O.csr_from_dense(a), g, eta, lam)
    kept = np.diff(ref.row_ptr)
    assert kept[::2].mean() > 0.5 * k or kept.max() > 0.5 * k   # some tiles dense
    assert kept.min() < 0.2 * k                                  # some tiles sparse
    _check_csr_equal(out, ref, transposed=transposed)
    assert ws.status()[0] == 0


@pytest.mark.parametrize("m,k,transposed", [(96, 256, True), (9, 9216, False)])
def test_prox_stash_boundary(C, m, k, transposed):
    """Tiles that keep exactly an eighth of their entries (written through
    the stash and copied into place) next to tiles that keep one entry more
    (written by the tile itself after the look-back), stored weights kept and
    dropped among them: bit-exact with the oracle. A row tile here is
    max(1, 8192 // k) rows; its stash holds tile_entries / 8 entries."""
    rows_per_tile = max(1, 8192 // k)
    cap = rows_per_tile * k // 8
    rng = np.random.default_rng(k)
    a = _sparse(rng, m, k, 0.02)
    g = np.zeros((m, k), F32)   # unstored entries with G = 0 are dropped
    eta, lam = 0.5, 0.1          # kept off the pattern iff |fl(0.5 G)| > 0.05
    tiles = (m + rows_per_tile - 1) // rows_per_tile
    for t in range(tiles):
        r0 = t * rows_per_tile
        blk = slice(r0, min(m, r0 + rows_per_tile))
        stored = a[blk] != 0
        n_stored = int(stored.sum())
        # every stored weight is kept (|w - 0| = |w| > 0.05 for these draws), so the tile keeps
        # n_stored + the unstored entries given a large G: cap, cap + 1, or fewer
        want = [cap, cap + 1, cap // 2][t % 3]
        free = np.flatnonzero(~stored.ravel())
        pick = rng.choice(free, size=max(0, want - n_stored), replace=False)
        gb = g[blk].ravel()
        gb[pick] = rng.choice([-1.0, 1.0], size=pick.size) * (1.0 + rng.random(pick.size))
        g[blk] = gb.reshape(g[blk].shape)
    a[(a != 0) & (np.abs(a) <= 0.05)] = 0.2   # stored weights all above the threshold
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(m, k, transposed=transposed)
    C.prox_update_compact(w, _dev(g), eta, lam, out, ws)
    ref = O.prox_update_compact(O.csr_from_dense(a), g, eta, lam)
    per_tile = np.add.reduceat(np.diff(ref.row_ptr), np.arange(0, m, rows_per_tile))
    assert (per_tile == cap).any() and (per_tile == cap + 1).any()
    _check_csr_equal(out, ref, transposed=transposed)
    assert ws.status()[0] == 0


@pytest.mark.parametrize("m,k", [(200, 333), (200, 320), (70, 4096)])
def test_prox_chain_of_steps_bit_exact(C, m, k):
    # several prox steps in a row (double-buffered), each fed the same G as the oracle
    rng = np.random.default_rng(21 + k)
    a = _sparse(rng, m, k, 0.2)
    ws = _ws(C, m, k, 1)
    bufs = [_gpu_csr(C, a, ws), C.CSR(m, k)]
    ref = O.csr_from_dense(a)
    for step in range(5):
        g = (rng.standard_normal((m, k)) * 0.3).astype(F32)
        C.prox_update_compact(bufs[step % 2], _dev(g), 0.05, 0.5, bufs[(step + 1) % 2], ws)
        ref = O.prox_update_compact(ref, g, 0.05, 0.5)
        _check_csr_equal(bufs[(step + 1) % 2], ref)


@pytest.mark.parametrize("eta,lam", [(0.0, 1e-4), (0.01, 0.0), (1e-3, 1e-38), (0.5, 1e30), (3.0, 1e-7),
                                     (1e-20, 1e-20)])
def test_fused_gradient_prox_threshold_edges(C, eta, lam):
    """The fused count pass decides an unstored entry by |G| > g*, the largest
    float with fl(eta*g*) <= fl(eta*lambda) (found on the host): the same keep
    decisions and values as weight_grad_dense (TF32) + prox_update_compact at
    eta = 0, lambda = 0, a subnormal threshold, a threshold above every
    product, and gradients scaled so that many products land on it."""
    m, k, n = 256, 512, 64
    rng = np.random.default_rng(int(1e3 * eta) + 7)
    a = _sparse(rng, m, k, 0.1) * F32(0.05)
    dy = _dev((rng.standard_normal((m, n)) * 1e-3).astype(F32))
    x = _dev(rng.standard_normal((k, n)).astype(F32))
    ws = _ws(C, m, k, n)
    w_in = _gpu_csr(C, a, ws, transposed=False)
    g = torch.zeros(m, k, device="cuda")
    C.weight_grad_dense(dy, x, g, ws, precision=C.CSRT_PREC_TF32)
    ref = C.CSR(m, k, transposed=True)
    C.prox_update_compact(w_in, g, eta, lam, ref, ws)
    out = C.CSR(m, k, transposed=True)
    C.weight_grad_prox_update(w_in, dy, x, eta, lam, out, ws)
    assert ws.status()[0] == 0
    (rp, ci, v), t = out.to_host()
    (rp2, ci2, v2), t2 = ref.to_host()
    np.testing.assert_array_equal(rp, rp2)
    np.testing.assert_array_equal(ci, ci2)
    np.testing.assert_array_equal(v.view(np.uint32), v2.view(np.uint32))
    for p_, q_ in zip(t, t2):
        np.testing.assert_array_equal(p_.view(np.uint32), q_.view(np.uint32))


@pytest.mark.parametrize("m,k,n,density,lam,transposed,zipf", [
    (300, 512, 64, 0.1, 0.05, True, False),
    (129, 320, 36, 0.2, 0.02, False, False),
    (200, 800, 128, 0.05, 0.03, True, False),
    (1000, 4096, 256, 0.15, 0.01, True, False),
    (64, 64, 4, 0.0, 0.0, True, False),
    (260, 9216, 64, 0.05, 0.02, True, False),
    (70, 16384, 32, 0.05, 0.02, False, False),
    # power-law rows (dense rows: every word past the prefetched weights) and
    # a fully dense input
    (400, 1024, 64, 0.3, 0.02, True, True),
    (160, 256, 32, 1.0, 0.05, True, False),
])
def test_fused_gradient_prox_matches_unfused(C, m, k, n, density, lam, transposed, zipf):
    """weight_grad_prox_update (G never written) gives the same bits as
    weight_grad_dense (TF32) followed by prox_update_compact."""
    rng = np.random.default_rng(m + k + n)
    a = _sparse(rng, m, k, density, zipf) * F32(0.05)
    dy = _dev((rng.standard_normal((m, n)) * 0.1).astype(F32))
    x = _dev(rng.standard_normal((k, n)).astype(F32))
    ws = _ws(C, m, k, n)
    w_in = _gpu_csr(C, a, ws, transposed=False)
    g = torch.zeros(m, k, device="cuda")
    C.weight_grad_dense(dy, x, g, ws, precision=C.CSRT_PREC_TF32)
    ref = C.CSR(m, k, transposed=transposed)
    C.prox_update_compact(w_in, g, 0.5, lam, ref, ws)
    out = C.CSR(m, k, transposed=transposed)
    C.weight_grad_prox_update(w_in, dy, x, 0.5, lam, out, ws)
    assert ws.status()[0] == 0
    (rp, ci, v), t = out.to_host()
    (rp2, ci2, v2), t2 = ref.to_host()
    np.testing.assert_array_equal(rp, rp2)
    np.testing.assert_array_equal(ci, ci2)
    np.testing.assert_array_equal(v.view(np.uint32), v2.view(np.uint32))
    if transposed:
        for p_, q_ in zip(t, t2):
            np.testing.assert_array_equal(p_.view(np.uint32), q_.view(np.uint32))
    # and against the oracle fed the same G
    refo = O.prox_update_compact(O.csr_from_dense(a), g.cpu().numpy(), 0.5, lam)
    np.testing.assert_array_equal(rp, refo.row_ptr)
    np.testing.assert_array_equal(ci, refo.col_idx)


def test_fused_gradient_prox_fallback_needs_scratch(C):
    rng = np.random.default_rng(1)
    m, k, n = 50, 40, 6                                   # too small for the tensor-core path
    a = _sparse(rng, m, k, 0.3)
    dy, x = _dev(rng.standard_normal((m, n)).astype(F32)), _dev(rng.standard_normal((k, n)).astype(F32))
    ws = _ws(C, m, k, n)
    w_in = _gpu_csr(C, a, ws)
    out = C.CSR(m, k)
    with pytest.raises(C.CsrtError):
        C.weight_grad_prox_update(w_in, dy, x, 0.1, 0.01, out, ws)
    g = torch.zeros(m, k, device="cuda")
    C.weight_grad_prox_update(w_in, dy, x, 0.1, 0.01, out, ws, g_scratch=g)
    ref = O.prox_update_compact(O.csr_from_dense(a), g.cpu().numpy(), 0.1, 0.01)
    (rp, ci, v), _ = out.to_host()
    np.testing.assert_array_equal(ci, ref.col_idx)
    np.testing.assert_array_equal(v.view(np.uint32), ref.val.view(np.uint32))


@pytest.mark.parametrize("m,k,transposed", [(256, 512, False), (256, 512, True), (300, 300, False),
                                            (129, 4100, True)])
def test_prox_capacity_overflow(C, m, k, transposed):
    """An output CSR too small for the prox result: the overflow and the needed
    nnz are reported, the row pointers are clamped and the stored prefix is the
    oracle's."""
    rng = np.random.default_rng(m + k + transposed)
    a = _sparse(rng, m, k, 0.2)
    g = rng.standard_normal((m, k)).astype(F32)
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws, transposed=False)
    ref = O.prox_update_compact(O.csr_from_dense(a), g, 0.5, 0.5)
    cap = ref.nnz // 3
    out = C.CSR(m, k, capacity=cap, transposed=transposed)
    C.prox_update_compact(w, _dev(g), 0.5, 0.5, out, ws)
    flags, required = ws.status()
    assert flags & C.CSRT_DEV_CAPACITY and required == ref.nnz
    rp = out.row_ptr.cpu().numpy()
    np.testing.assert_array_equal(rp, np.minimum(ref.row_ptr, cap))
    np.testing.assert_array_equal(out.col_idx.cpu().numpy()[:cap], ref.col_idx[:cap])
    np.testing.assert_array_equal(out.val.cpu().numpy()[:cap].view(np.uint32), ref.val[:cap].view(np.uint32))
    ws.clear_status()


def test_prox_nan_is_dropped_and_flagged(C):
    a = np.array([[1.0, 0.0, 2.0, 0.0]], dtype=F32)
    g = np.array([[np.nan, 1.0, 0.0, np.nan]], dtype=F32)
    ws = _ws(C, 1, 4, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(1, 4)
    C.prox_update_compact(w, _dev(g), 0.5, 0.25, out, ws)
    (rp, ci, v), _ = out.to_host()
    assert ci.tolist() == [1, 2]
    assert ws.status()[0] & C.CSRT_DEV_NONFINITE


def test_debias_bit_exact_and_pattern_fixed(C):
    rng = np.random.default_rng(5)
    m, k = 120, 90
    a = _sparse(rng, m, k, 0.3)
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    ref = O.csr_from_dense(a)
    g = rng.standard_normal(ref.nnz).astype(F32)
    g[0] = ref.val[0] / F32(0.25)
    before = w.to_host()
    C.debias_update(w, _dev(g), 0.25)
    (rp, ci, v), t = w.to_host()
    out = O.debias_update(ref, g, 0.25)
    np.testing.assert_array_equal(rp, before[0][0])
    np.testing.assert_array_equal(ci, before[0][1])
    np.testing.assert_array_equal(v.view(np.uint32), out.val.view(np.uint32))
    assert v[0] == 0.0
    np.testing.assert_array_equal(t[0], before[1][0])
    np.testing.assert_array_equal(t[1], before[1][1])
    np.testing.assert_array_equal(t[2][t[3]].view(np.uint32), v.view(np.uint32))


# --- glue ----------------------------------------------------------------------

def test_glue_layers(C):
    rng = np.random.default_rng(9)
    c, b, h, w, k = 3, 4, 12, 10, 5
    x = rng.standard_normal((c, b, h, w)).astype(F32)
    ho, wo = h - k + 1, w - k + 1
    cols = torch.zeros(c * k * k, b * ho * wo, device="cuda")
    C.im2col(_dev(x.reshape(c, -1)), c, b, h, w, k, cols)
    np.testing.assert_array_equal(cols.cpu().numpy(), O.im2col(x, k))
    dcols = rng.standard_normal((c * k * k, b * ho * wo)).astype(F32)
    dx = torch.zeros(c, b * h * w, device="cuda")
    C.col2im(_dev(dcols), c, b, h, w, k, dx)
    assert_close(dx.cpu().numpy().reshape(c, b, h, w), O.col2im(dcols, c, b, h, w, k), what="col2im")
    xp = rng.standard_normal((c, b, 8, 6)).astype(F32)
    xp[0, 0, 0, :2] = 7.0                                   # a tie: first maximum wins
    y = torch.zeros(c, b * 4 * 3, device="cuda")
    idx = torch.zeros(c * b * 12, dtype=torch.int8, device="cuda")
    C.maxpool2_fwd(_dev(xp.reshape(c, -1)), c, b, 8, 6, y, idx)
    ry, ridx = O.maxpool2_fwd(xp)
    np.testing.assert_array_equal(y.cpu().numpy().reshape(ry.shape), ry)
    np.testing.assert_array_equal(idx.cpu().numpy().reshape(ridx.shape), ridx)
    dyp = rng.standard_normal(ry.shape).astype(F32)
    dxp = torch.zeros(c, b * 48, device="cuda")
    C.maxpool2_bwd(_dev(dyp.reshape(c, -1)), idx, c, b, 8, 6, dxp)
    np.testing.assert_array_equal(dxp.cpu().numpy().reshape(xp.shape), O.maxpool2_bwd(dyp, ridx))
    xf = torch.zeros(c * 48, b, device="cuda")
    C.flatten(_dev(xp.reshape(c, -1)), c, b, 48, xf)
    np.testing.assert_array_equal(xf.cpu().numpy(), O.flatten_cnhw(xp))
    back = torch.zeros(c, b * 48, device="cuda")
    C.unflatten(xf, c, b, 48, back)
    np.testing.assert_array_equal(back.cpu().numpy().reshape(xp.shape), xp)


def test_bias_relu_softmax(C):
    rng = np.random.default_rng(10)
    m, n = 37, 70
    y0 = rng.standard_normal((m, n)).astype(F32)
    bias = rng.standard_normal(m).astype(F32)
    y = _dev(y0)
    C.bias_act_fwd(y, _dev(bias), True)
    np.testing.assert_array_equal(y.cpu().numpy(), np.maximum(y0 + bias[:, None], 0).astype(F32))
    d0 = rng.standard_normal((m, n)).astype(F32)
    d = _dev(d0)
    C.relu_bwd(d, y)
    np.testing.assert_array_equal(d.cpu().numpy(), np.where(y.cpu().numpy() > 0, d0, 0))
    b = _dev(bias)
    gb = torch.zeros(m, device="cuda")
    C.bias_grad_sgd(d, b, 0.1, gb)
    ref_gb = d.cpu().numpy().astype(np.float64).sum(axis=1)
    assert_close(gb.cpu().numpy(), ref_gb, np.abs(d.cpu().numpy()).sum(axis=1), n, what="bias grad")
    np.testing.assert_array_equal(b.cpu().numpy(), (bias - F32(0.1) * gb.cpu().numpy()).astype(F32))
    for classes in (10, 1000):
        z = rng.standard_normal((classes, n)).astype(F32) * 3
        lab = rng.integers(0, classes, n).astype(np.int32)
        dz = torch.zeros(classes, n, device="cuda")
        loss = torch.zeros(n + 1, device="cuda")
        C.softmax_xent(_dev(z), _dev(lab), dz, loss)
        rl, rdz = O.softmax_xent(z, lab)
        assert abs(loss[0].item() - rl) <= 1e-5 * max(1, abs(rl))
        assert_close(dz.cpu().numpy(), rdz, rtol=1e-4, atol=1e-7, what="softmax dz")


# --- Prox-RMSProp (Algorithm 1) and Prox-ADAM (Algorithm 2) -----------------

def test_adaptive_hand_cases_on_gpu(C):
    with open(os.path.join(GOLD, "adaptive_prox_cases.json")) as f:
        d = json.load(f)

    def run(cases, adam, t=1):
        k = len(cases)
        w0 = np.array([[c["w"] for c in cases]], dtype=F32)
        g = _dev(np.array([[c["g"] for c in cases]], dtype=F32))
        v = _dev(np.array([[c["v"] for c in cases]], dtype=F32))
        ws = _ws(C, 1, k, 1)
        w = _gpu_csr(C, w0, ws)
        out = C.CSR(1, k)
        if adam:
            m = _dev(np.array([[c["m"] for c in cases]], dtype=F32))
            c0 = cases[0]
            C.prox_adam_update_compact(w, g, m, v, t, d["eta"], d["lambda"], c0["beta1"], c0["beta2"], c0["eps"],
                                       out, ws)
            assert m.cpu().numpy()[0].tolist() == [c["m_new"] for c in cases]
        else:
            c0 = cases[0]
            C.prox_rmsprop_update_compact(w, g, v, d["eta"], d["lambda"], c0["beta"], c0["eps"], out, ws)
        assert v.cpu().numpy()[0].tolist() == [c["v_new"] for c in cases]
        (rp, ci, vals), _ = out.to_host()
        dense = csr_dense(rp, ci, vals, 1, k)[0]
        for j, c in enumerate(cases):
            assert (dense[j] if dense[j] != 0 else None) == c["w_new"], c
        assert ws.status()[0] == 0

    run(d["rmsprop"], adam=False)
    run([c for c in d["adam"] if c["t"] == 1], adam=True, t=1)
    run([c for c in d["adam"] if c["t"] == 2], adam=True, t=2)


@pytest.mark.parametrize("opt", ["adam", "rmsprop"])
@pytest.mark.parametrize("m,k,density", [
    (300, 784, 0.1),        # row tiles
    (37, 4099, 0.3),        # K % 4 != 0: flat tiles
    (4097, 3, 0.6),
    (3, 16384, 0.02),       # the longest row-tile rows
    (2, 16388, 0.02),       # beyond them: flat tiles
    (1000, 4096, 0.15),     # the classifier head's last layer
])
def test_adaptive_prox_chain_bit_exact(C, opt, m, k, density):
    """Three adaptive prox steps in a row (double-buffered CSR, moments kept
    on the GPU), each against the oracle fed the same G and the oracle's own
    moments: the CSR, its transposed arrays and the moments bit for bit."""
    rng = np.random.default_rng(m + 3 * k)
    a = _sparse(rng, m, k, density) * F32(0.1)
    ws = _ws(C, m, k, 1)
    bufs = [_gpu_csr(C, a, ws), C.CSR(m, k)]
    mom = [torch.zeros(m, k, device="cuda"), torch.zeros(m, k, device="cuda")]
    ref = O.csr_from_dense(a)
    rm = np.zeros((m, k), dtype=F32)
    rv = np.zeros((m, k), dtype=F32)
    eta, lam = 0.01, 0.5
    for t in range(1, 4):
        g = (rng.standard_normal((m, k)) * 0.3).astype(F32)
        if opt == "adam":
            C.prox_adam_update_compact(bufs[(t - 1) % 2], _dev(g), mom[0], mom[1], t, eta, lam, 0.9, 0.999, 1e-8,
                                       bufs[t % 2], ws)
            ref, rm, rv = O.prox_adam_update_compact(ref, g, rm, rv, t, eta, lam, 0.9, 0.999, 1e-8)
            np.testing.assert_array_equal(mom[0].cpu().numpy().view(np.uint32), rm.view(np.uint32))
        else:
            C.prox_rmsprop_update_compact(bufs[(t - 1) % 2], _dev(g), mom[1], eta, lam, 0.9, 1e-8, bufs[t % 2], ws)
            ref, rv = O.prox_rmsprop_update_compact(ref, g, rv, eta, lam, 0.9, 1e-8)
        np.testing.assert_array_equal(mom[1].cpu().numpy().view(np.uint32), rv.view(np.uint32))
        _check_csr_equal(bufs[t % 2], ref)
        assert ref.nnz > 0
    assert ws.status()[0] == 0


def test_adaptive_prox_unaligned_moments(C):
    # moments that are not 16-byte aligned take the flat tiles: same result
    m, k = 64, 256
    rng = np.random.default_rng(3)
    a = _sparse(rng, m, k, 0.2)
    g = (rng.standard_normal((m, k)) * 0.3).astype(F32)
    ws = _ws(C, m, k, 1)
    w = _gpu_csr(C, a, ws)
    store = torch.zeros(2 * m * k + 2, device="cuda")
    mm, vv = store[1:1 + m * k], store[m * k + 2:]
    out = C.CSR(m, k)
    C.prox_adam_update_compact(w, _dev(g), mm, vv, 1, 0.01, 0.5, 0.9, 0.999, 1e-8, out, ws)
    ref, rm, rv = O.prox_adam_update_compact(O.csr_from_dense(a), g, np.zeros((m, k), F32), np.zeros((m, k), F32),
                                             1, 0.01, 0.5, 0.9, 0.999, 1e-8)
    _check_csr_equal(out, ref)
    np.testing.assert_array_equal(mm.cpu().numpy().view(np.uint32), rm.reshape(-1).view(np.uint32))
    np.testing.assert_array_equal(vv.cpu().numpy().view(np.uint32), rv.reshape(-1).view(np.uint32))


def test_adaptive_prox_nan_and_arguments(C):
    a = np.array([[1.0, 0.0, 2.0, 0.0]], dtype=F32)
    g = _dev(np.array([[np.nan, 1.0, 0.0, 1.0]], dtype=F32))
    ws = _ws(C, 1, 4, 1)
    w = _gpu_csr(C, a, ws)
    out = C.CSR(1, 4)
    m, v = torch.zeros(1, 4, device="cuda"), torch.zeros(1, 4, device="cuda")
    C.prox_adam_update_compact(w, g, m, v, 1, 0.5, 0.25, 0.9, 0.999, 1e-8, out, ws)
    (rp, ci, vals), _ = out.to_host()
    assert 0 not in ci.tolist()                       # the NaN direction drops its entry
    assert ws.status()[0] & C.CSRT_DEV_NONFINITE
    lib = C.lib()
    bad = [
        lambda: lib.prox_adam_update_compact(w.struct, C._ptr(g), C._ptr(m), C._ptr(v), 0, 0.5, 0.25, 0.9, 0.999,
                                             1e-8, out.struct, ws.ptr, ws.nbytes, None),          # t = 0
        lambda: lib.prox_adam_update_compact(w.struct, C._ptr(g), C._ptr(m), C._ptr(v), 1, 0.5, 0.25, 1.0, 0.999,
                                             1e-8, out.struct, ws.ptr, ws.nbytes, None),          # beta1 = 1
        lambda: lib.prox_rmsprop_update_compact(w.struct, C._ptr(g), C._ptr(v), 0.5, 0.25, 0.9, 0.0, out.struct,
                                                ws.ptr, ws.nbytes, None),                         # eps = 0
        lambda: lib.prox_rmsprop_update_compact(w.struct, C._ptr(g), C._ptr(g), 0.5, 0.25, 0.9, 1e-8, out.struct,
                                                ws.ptr, ws.nbytes, None),                         # v aliases G
    ]
    for call in bad:
        assert call() == C.CSRT_ERR_ARG


# --- convolution with CSR filters, input read in place -----------------------

@pytest.mark.parametrize("cout,cin,b,h,w,k,density,relu", [
    (20, 1, 3, 28, 28, 5, 158 / 500, False),      # LeNet-5 conv1 at the SpC density of the layer table
    (50, 20, 2, 12, 12, 5, 2101 / 25000, False),  # conv2
    (7, 3, 2, 7, 9, 3, 0.5, True),                # ragged shapes, ReLU
    (4, 2, 1, 5, 5, 5, 0.0, True),                # no stored taps: bias (and ReLU) only
    (3, 60, 1, 6, 6, 5, 1.0, False),              # 1500 taps per filter: two staging rounds
])
def test_conv2d_sparse_fwd_against_oracle(C, cout, cin, b, h, w, k, density, relu):
    rng = np.random.default_rng(cout * cin + h)
    wt = _sparse(rng, cout, cin * k * k, density)
    x = rng.standard_normal((cin, b, h, w)).astype(F32)
    bias = rng.standard_normal(cout).astype(F32)
    ws = _ws(C, cout, cin * k * k, 1)
    W = _gpu_csr(C, wt, ws, transposed=False)
    ho, wo = h - k + 1, w - k + 1
    y = torch.full((cout, b * ho * wo), float("nan"), device="cuda")
    C.conv2d_sparse_fwd(W, _dev(x.reshape(cin, -1)), cin, b, h, w, k, _dev(bias), relu, y)
    ref_w = O.csr_from_dense(wt)
    cols = O.im2col(x, k)
    pre = O.spmm_fwd(ref_w, cols) + bias.astype(np.float64)[:, None]
    ref = np.maximum(pre, 0.0) if relu else pre
    bound = O.spmm_fwd(O.csr_abs(ref_w), np.abs(cols)) + np.abs(bias.astype(np.float64))[:, None]
    assert_close(y.cpu().numpy(), ref, bound, (np.diff(ref_w.row_ptr) + 1)[:, None], what="conv2d_sparse_fwd")


# --- failure detection: bounded waits give up and report ---------------------

def test_bounded_waits_give_up_and_report(C):
    """The look-back spin and the mbarrier wait, run against a predecessor and
    a barrier that never arrive, give up, set CSRT_DEV_TIMEOUT and return;
    the context stays usable for the next product."""
    import time
    ws = _ws(C, 64, 64, 64)
    ws.clear_status()
    assert ws.status()[0] == 0
    t0 = time.time()
    C.check_bounded_waits(ws)
    flags, _ = ws.status()
    assert flags & C.CSRT_DEV_TIMEOUT
    assert time.time() - t0 < 60
    ws.clear_status()
    rng = np.random.default_rng(2)
    a = _sparse(rng, 64, 64, 0.2)
    x = rng.standard_normal((64, 16)).astype(F32)
    w = _gpu_csr(C, a, ws)
    y = torch.zeros(64, 16, device="cuda")
    C.spmm_fwd(w, _dev(x), y, ws)
    ref = O.csr_from_dense(a)
    assert_close(y.cpu().numpy(), O.spmm_fwd(ref, x), O.spmm_fwd(O.csr_abs(ref), np.abs(x)),
                 np.diff(ref.row_ptr)[:, None], what="spmm after the timed-out waits")
    assert ws.status()[0] == 0


@pytest.mark.parametrize("m,k,n,density,mix", [(256, 512, 64, 0.05, False), (1000, 4096, 256, 0.05, False),
                                               (512, 2048, 128, 0.05, True), (300, 1024, 32, 0.02, True),
                                               (128, 9216, 256, 0.08, True)])
def test_fused_gradient_prox_sparse_and_dense_words(C, m, k, n, density, mix):
    """The write pass stores a 32-column word whose 32 rows keep few entries
    (at most 96) by per-row compaction and one entry per lane, and other words
    by the row walk. Small gradients keep little more than the stored weights
    (sparse words); with `mix`, alternate 32-row bands get large gradients
    (dense words), so both forms run in one call. Bit-identical to
    weight_grad_dense (TF32) + prox_update_compact, transposed copy included."""
    rng = np.random.default_rng(m + k + n)
    a = _sparse(rng, m, k, density) * F32(0.05)
    scale = np.full((m, 1), 1e-5, dtype=F32)
    if mix:
        scale[(np.arange(m) // 32) % 2 == 1] = F32(0.1)
    dy = _dev((rng.standard_normal((m, n)) * scale).astype(F32))
    x = _dev(rng.standard_normal((k, n)).astype(F32))
    ws = _ws(C, m, k, n)
    w_in = _gpu_csr(C, a, ws, transposed=False)
    g = torch.zeros(m, k, device="cuda")
    C.weight_grad_dense(dy, x, g, ws, precision=C.CSRT_PREC_TF32)
    ref = C.CSR(m, k, transposed=True)
    C.prox_update_compact(w_in, g, 0.5, 2e-3, ref, ws)
    out = C.CSR(m, k, transposed=True)
    C.weight_grad_prox_update(w_in, dy, x, 0.5, 2e-3, out, ws)
    assert ws.status()[0] == 0
    (rp, ci, v), t = out.to_host()
    (rp2, ci2, v2), t2 = ref.to_host()
    kept = np.diff(rp.astype(np.int64))
    assert kept.min() < 0.1 * k   # sparse rows present
    if mix:
        assert kept.max() > 0.5 * k   # and dense ones
    np.testing.assert_array_equal(rp, rp2)
    np.testing.assert_array_equal(ci, ci2)
    np.testing.assert_array_equal(v.view(np.uint32), v2.view(np.uint32))
    for p_, q_ in zip(t, t2):
        np.testing.assert_array_equal(p_.view(np.uint32), q_.view(np.uint32))


@pytest.mark.parametrize("dy_scale", [0.1, 1e-5])
@pytest.mark.parametrize("transposed", [False, True])
def test_fused_gradient_prox_capacity_overflow(C, transposed, dy_scale):
    """An output CSR too small for the fused op's result: the overflow and the
    needed nnz are reported, the row pointers are clamped, and the stored
    prefix equals the unfused result's (the transposed copy, when asked for,
    writes only inside the capacity)."""
    m, k, n = 256, 512, 64
    rng = np.random.default_rng(9)
    a = _sparse(rng, m, k, 0.1 if dy_scale > 1e-3 else 0.05) * F32(0.05)   # dense words, or sparse ones
    dy = _dev((rng.standard_normal((m, n)) * dy_scale).astype(F32))
    x = _dev(rng.standard_normal((k, n)).astype(F32))
    ws = _ws(C, m, k, n)
    w_in = _gpu_csr(C, a, ws, transposed=False)
    g = torch.zeros(m, k, device="cuda")
    C.weight_grad_dense(dy, x, g, ws, precision=C.CSRT_PREC_TF32)
    ref = C.CSR(m, k, transposed=False)
    C.prox_update_compact(w_in, g, 0.5, 0.01, ref, ws)
    (rp_ref, ci_ref, v_ref), _ = ref.to_host()
    nnz = int(rp_ref[-1])
    assert ws.status()[0] == 0
    cap = nnz // 3
    out = C.CSR(m, k, capacity=cap, transposed=transposed)
    C.weight_grad_prox_update(w_in, dy, x, 0.5, 0.01, out, ws)
    flags, required = ws.status()
    assert flags & C.CSRT_DEV_CAPACITY and required == nnz
    rp = out.row_ptr.cpu().numpy()
    assert (np.diff(rp) >= 0).all() and rp[-1] == cap
    np.testing.assert_array_equal(rp, np.minimum(rp_ref, cap))
    np.testing.assert_array_equal(out.col_idx.cpu().numpy()[:cap], ci_ref[:cap])
    np.testing.assert_array_equal(out.val.cpu().numpy()[:cap].view(np.uint32), v_ref[:cap].view(np.uint32))
    ws.clear_status()
