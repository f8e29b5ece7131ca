"""csrt_validate_csr: valid CSRs (built by the library, after prox steps,
empty rows and matrices) pass; CSRs corrupted on the host side (a column out
of range, unsorted or repeated columns, non-monotone or out-of-capacity row
pointers, a wrong transposed position, value or row) are reported with the
first broken row, and nothing is read out of range meanwhile."""

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import csrtrain
    csrtrain.lib()
    return csrtrain


def _build(C, m, k, density, seed=0, transposed=True, capacity=None):
    from paper_1905_07931_gb300 import synth
    rng = np.random.default_rng(seed)
    a = synth.masked_weights(rng, m, k, density)
    if m > 3:
        a[3, :] = 0.0   # an empty row
    ws = C.Workspace(max(m, 1), max(k, 1), 1)
    w = C.CSR(m, k, capacity=capacity, transposed=transposed)
    C.csr_from_dense(torch.from_numpy(a).cuda(), w, ws)
    return w, ws


@pytest.mark.parametrize("m,k,density,transposed", [(300, 784, 0.1, True), (1, 1, 1.0, True), (64, 64, 0.0, True),
                                                     (2000, 300, 0.3, True), (129, 257, 0.2, False)])
def test_valid_csrs_pass(C, m, k, density, transposed):
    w, ws = _build(C, m, k, density, transposed=transposed)
    assert C.validate_csr(w, ws) is None
    assert ws.status()[0] == 0


def test_prox_output_passes(C):
    w, ws = _build(C, 500, 800, 0.1)
    out = C.CSR(500, 800)
    g = torch.randn(500, 800, device="cuda")
    C.prox_update_compact(w, g, 0.1, 0.5, out, ws)
    assert C.validate_csr(out, ws) is None
    assert ws.status()[0] == 0


def test_empty_shapes_pass(C):
    ws = C.Workspace(4, 4, 1)
    for m, k in [(0, 5), (5, 0), (0, 0)]:
        w = C.CSR(m, k, capacity=0)
        assert C.validate_csr(w, ws) is None
    assert ws.status()[0] == 0


def _corrupt_and_check(C, w, ws, expect_row):
    ws.clear_status()
    row = C.validate_csr(w, ws)
    flags, _ = ws.status()
    assert flags & C.CSRT_DEV_INVALID, flags
    assert row == expect_row, (row, expect_row)
    ws.clear_status()
    assert C.validate_csr(w, ws) == expect_row   # the check is repeatable
    ws.clear_status()


def test_corrupted_rows_are_reported(C):
    m, k = 300, 784
    w, ws = _build(C, m, k, 0.1, seed=1, transposed=False)
    rp = w.row_ptr.cpu().numpy()

    col = w.col_idx.clone()
    w.col_idx[rp[10]] = k                        # a column past the matrix
    _corrupt_and_check(C, w, ws, 10)
    w.col_idx.copy_(col)

    w.col_idx[rp[20]], w.col_idx[rp[20] + 1] = col[rp[20] + 1], col[rp[20]]   # unsorted
    _corrupt_and_check(C, w, ws, 20)
    w.col_idx.copy_(col)

    w.col_idx[rp[30] + 1] = col[rp[30]]          # a repeated column
    _corrupt_and_check(C, w, ws, 30)
    w.col_idx.copy_(col)

    w.col_idx[rp[40]] = -1                       # a negative column
    _corrupt_and_check(C, w, ws, 40)
    w.col_idx.copy_(col)
    assert C.validate_csr(w, ws) is None


def test_corrupted_row_pointers_are_reported(C):
    m, k = 300, 784
    w, ws = _build(C, m, k, 0.1, seed=2, transposed=False, capacity=300 * 784)
    rp = w.row_ptr.clone()

    w.row_ptr[50] = rp[52]                       # row 49 ends after row 50 does: not monotone
    _corrupt_and_check(C, w, ws, 49)
    w.row_ptr.copy_(rp)

    w.row_ptr[m] = 2 ** 30                       # more entries than the capacity: never dereferenced
    _corrupt_and_check(C, w, ws, m - 1)
    w.row_ptr.copy_(rp)

    w.row_ptr[0] = 1                             # the first row pointer is not 0
    _corrupt_and_check(C, w, ws, 0)
    w.row_ptr.copy_(rp)

    w.row_ptr[7] = -5                            # a negative row pointer
    _corrupt_and_check(C, w, ws, 6)
    w.row_ptr.copy_(rp)
    assert C.validate_csr(w, ws) is None


def test_corrupted_transposed_copy_is_reported(C):
    m, k = 300, 784
    w, ws = _build(C, m, k, 0.1, seed=3)
    rp = w.row_ptr.cpu().numpy()
    saved = [t.clone() for t in (w.t_pos, w.t_val, w.t_col_idx, w.t_row_ptr)]

    w.t_pos[rp[12]] = w.t_pos[rp[12]] + 1        # an entry points at its neighbour
    _corrupt_and_check(C, w, ws, m + k + 1 + 12)
    w.t_pos.copy_(saved[0])

    w.t_val[w.t_pos[rp[15]]] += 1.0              # a transposed value differs
    _corrupt_and_check(C, w, ws, m + k + 1 + 15)
    w.t_val.copy_(saved[1])

    p = int(w.t_pos[rp[18]])
    w.t_col_idx[p] = 17                          # a transposed entry names the wrong row
    first = C.validate_csr(w, ws)                # the column's rows are no longer ascending, or the row differs
    assert first is not None and ws.status()[0] & C.CSRT_DEV_INVALID
    ws.clear_status()
    w.t_col_idx.copy_(saved[2])

    w.t_pos[rp[25]] = 2 ** 30                    # a position past the capacity: never dereferenced
    _corrupt_and_check(C, w, ws, m + k + 1 + 25)
    w.t_pos.copy_(saved[0])

    w.t_row_ptr[k] = w.t_row_ptr[k] - 1          # entry counts differ
    first = C.validate_csr(w, ws)
    assert first is not None and ws.status()[0] & C.CSRT_DEV_INVALID
    ws.clear_status()
    w.t_row_ptr.copy_(saved[3])
    assert C.validate_csr(w, ws) is None
    assert ws.status()[0] == 0
