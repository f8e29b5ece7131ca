"""Error behaviour of the C ABI on the host: every call checks its arguments
before it touches the GPU and returns CSRT_ERR_ARG with a message (nothing
enqueued). Each case below fails a host-side check, so no device memory is
read: the non-NULL pointers are placeholders that are never dereferenced."""

import ctypes

import pytest

FAKE = ctypes.c_void_p(256)   # non-NULL, 16-byte aligned, never dereferenced


@pytest.fixture(scope="module")
def C():
    from paper_1905_07931_gb300 import build
    build.build()
    from paper_1905_07931_gb300 import csrtrain
    csrtrain.lib()
    return csrtrain


def _csr(C, rows=8, cols=8, capacity=64, transposed=False, base=256):
    p = [ctypes.c_void_p(base + 4096 * i) for i in range(7)]   # distinct placeholders per array
    t = p[3:] if transposed else [None] * 4
    return C.csrt_csr(rows, cols, capacity, p[0], p[1], p[2], *t)


def _expect(C, rc, fragment):
    assert rc == C.CSRT_ERR_ARG, rc
    msg = C.lib().csrt_last_error().decode()
    assert fragment in msg, msg


def test_sparse_products_reject_bad_arguments(C):
    L = C.lib()
    w = _csr(C)
    ws, nbytes = FAKE, ctypes.c_size_t(1 << 20)
    _expect(C, L.spmm_fwd(None, FAKE, 4, FAKE, ws, nbytes, None), "NULL")
    _expect(C, L.spmm_fwd(ctypes.byref(_csr(C, rows=-1)), FAKE, 4, FAKE, ws, nbytes, None), "negative shape")
    _expect(C, L.spmm_fwd(ctypes.byref(w), FAKE, -1, FAKE, ws, nbytes, None), "n < 0")
    _expect(C, L.spmm_fwd(ctypes.byref(w), None, 4, None, ws, nbytes, None), "X or Y is NULL")
    _expect(C, L.spmm_fwd(ctypes.byref(_csr(C, capacity=1 << 31)), FAKE, 4, FAKE, ws, nbytes, None), "capacity")
    _expect(C, L.spmm_bwd_t(ctypes.byref(w), FAKE, 4, FAKE, ws, nbytes, None), "transposed arrays not set")
    _expect(C, L.spmm_fwd_bias_act(ctypes.byref(w), FAKE, -2, FAKE, 1, FAKE, ws, nbytes, None), "n < 0")
    _expect(C, L.spmm_bwd_t_relu(ctypes.byref(w), FAKE, 4, FAKE, FAKE, ws, nbytes, None), "transposed arrays not set")
    _expect(C, L.spmm_fwd_noalloc(ctypes.byref(w), FAKE, 5000, FAKE, None), "exceeds the maximum")
    _expect(C, L.weight_grad_sddmm(ctypes.byref(w), FAKE, FAKE, -3, FAKE, ws, nbytes, None), "n < 0")
    _expect(C, L.debias_update(ctypes.byref(w), FAKE, ctypes.c_float(-1.0), None), "eta")


def test_gradients_and_prox_reject_bad_arguments(C):
    L = C.lib()
    w_in, w_out = _csr(C), _csr(C, base=1 << 20)
    nbytes = ctypes.c_size_t(1 << 20)
    f = ctypes.c_float
    _expect(C, L.weight_grad_dense(FAKE, FAKE, -1, 8, 4, FAKE, 1, FAKE, nbytes, None), "negative size")
    _expect(C, L.weight_grad_dense(FAKE, FAKE, 8, 8, 4, FAKE, 7, FAKE, nbytes, None), "unknown precision")
    _expect(C, L.prox_update_compact(ctypes.byref(w_in), FAKE, f(0.1), f(0.1), ctypes.byref(w_in), FAKE, nbytes,
                                     None), "alias")
    _expect(C, L.prox_update_compact(ctypes.byref(w_in), FAKE, f(-0.1), f(0.1), ctypes.byref(w_out), FAKE, nbytes,
                                     None), "finite and >= 0")
    other = _csr(C, cols=9, base=1 << 20)
    _expect(C, L.prox_update_compact(ctypes.byref(w_in), FAKE, f(0.1), f(0.1), ctypes.byref(other), FAKE, nbytes,
                                     None), "shapes differ")
    _expect(C, L.weight_grad_prox_update(ctypes.byref(w_in), FAKE, FAKE, 4, f(0.1), f(0.1), 5, None,
                                         ctypes.byref(w_out), FAKE, nbytes, None), "unknown precision")
    _expect(C, L.prox_adam_update_compact(ctypes.byref(w_in), FAKE, ctypes.c_void_p(512), ctypes.c_void_p(768), 0,
                                          f(0.1), f(0.1), f(0.9), f(0.999), f(1e-8), ctypes.byref(w_out), FAKE,
                                          nbytes, None), "step counter")
    _expect(C, L.prox_rmsprop_update_compact(ctypes.byref(w_in), FAKE, ctypes.c_void_p(512), f(0.1), f(0.1),
                                             f(1.5), f(1e-8), ctypes.byref(w_out), FAKE, nbytes, None), "beta")
    _expect(C, L.csr_from_dense(FAKE, 8, 9, ctypes.byref(w_out), FAKE, nbytes, None), "shape differs")
    _expect(C, L.csrt_validate_csr(None, FAKE, nbytes, None), "NULL")


def test_glue_rejects_bad_shapes(C):
    L = C.lib()
    _expect(C, L.csrt_softmax_xent(FAKE, FAKE, 0, 4, FAKE, FAKE, None), "bad size")
    _expect(C, L.csrt_im2col(FAKE, 1, 2, 3, 3, 5, FAKE, None), "bad shape")
    _expect(C, L.csrt_maxpool2_fwd(FAKE, 1, 2, 3, 4, FAKE, FAKE, None), "bad shape")
