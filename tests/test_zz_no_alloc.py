"""spmm_fwd_noalloc: the forward product for callers that cannot allocate.

Those callers (code inside a framework that owns every device allocation, or
a serving loop that may not allocate) get the same product as spmm_fwd, with
the scratch for split rows taken from a fixed array inside the library. This
test calls the entry point directly through the C ABI, twice in a row on
shapes whose rows are split between work units (so the scratch is used and
its contents from the first call are left behind for the second), and checks
the output against spmm_fwd with a caller workspace, and that the library's
own status word reports no bounded wait that gave up. It lives in a file that
pytest collects last so that a stop-at-first-failure run has already run
every other test; it also passes on its own in a fresh process.
"""

import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_noalloc_matches_spmm_fwd_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import csrtrain as C
    from paper_1905_07931_gb300 import synth

    lib = C.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    flags = ctypes.c_int32(-1)
    assert lib.spmm_fwd_noalloc_status(ctypes.byref(flags), 1, stream) == C.CSRT_OK
    for (m, k, n, zipf) in [(700, 900, 96, True), (300, 784, 256, False), (64, 20000, 1, False),
                            (700, 900, 32, True)]:
        rng = np.random.default_rng(m + n)
        w = synth.masked_weights(rng, m, k, 0.1, zipf=zipf)
        ws = C.Workspace(m, k, n)
        W = C.CSR(m, k, transposed=False)
        C.csr_from_dense(torch.from_numpy(w).cuda(), W, ws)
        ref = torch.zeros(m, n, device="cuda")
        for call in range(2):
            x = torch.from_numpy(rng.standard_normal((k, n)).astype(np.float32)).cuda()
            C.spmm_fwd(W, x, ref, ws)
            y = torch.full((m, n), float("nan"), device="cuda")
            C.launch_count(reset=True)
            rc = lib.spmm_fwd_noalloc(W.struct, ctypes.c_void_p(x.data_ptr()), n,
                                      ctypes.c_void_p(y.data_ptr()), stream)
            assert rc == C.CSRT_OK, lib.csrt_last_error()
            # the product kernel and the fix-up kernel: rows are split between
            # work units, so the static scratch carries partial sums
            assert C.launch_count() == 2
            torch.cuda.synchronize()
            got, exp = y.cpu().numpy(), ref.cpu().numpy()
            # Same kernels and partition as spmm_fwd. Where spmm_fwd completes
            # a shared row inside the product kernel (wide n), it adds the
            # units' carries in unit order, as the fix-up kernel does here:
            # identical bits (well inside the 1e-4 parity tolerance).
            np.testing.assert_array_equal(got.view(np.uint32), exp.view(np.uint32))
        assert ws.status()[0] == 0
    # no bounded wait gave up in any call above
    assert lib.spmm_fwd_noalloc_status(ctypes.byref(flags), 0, stream) == C.CSRT_OK
    assert flags.value == 0


def test_noalloc_rejects_shapes_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import csrtrain as C
    W = C.CSR(64, 64, transposed=False)
    n = 4100                                    # the documented maximum is 4096 columns
    x = torch.zeros(64, n, device="cuda")
    y = torch.zeros(64, n, device="cuda")
    rc = C.lib().spmm_fwd_noalloc(W.struct, ctypes.c_void_p(x.data_ptr()), n, ctypes.c_void_p(y.data_ptr()),
                                  ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == C.CSRT_ERR_ARG
    assert b"static scratch" in C.lib().csrt_last_error()
