"""ctypes binding of libcsrtrain.so (include/csrtrain.h).

Argument marshalling only: every function takes torch tensors that already
live on the GPU, checks dtype / shape / contiguity, and passes raw device
pointers and sizes to the C ABI on the current (or given) CUDA stream. All
arithmetic runs in the CUDA library; there is no CPU fallback, and loading
fails loudly if the library has not been built.
"""

from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int8, c_int32, c_int64, c_size_t, c_void_p

import torch

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libcsrtrain.so")

CSRT_OK, CSRT_ERR_ARG, CSRT_ERR_CUDA, CSRT_ERR_WORKSPACE = 0, 1, 2, 3
CSRT_DEV_CAPACITY, CSRT_DEV_TIMEOUT, CSRT_DEV_NONFINITE, CSRT_DEV_INVALID = 1, 2, 4, 8
CSRT_PREC_FP32, CSRT_PREC_TF32 = 0, 1


class csrt_csr(ctypes.Structure):
    _fields_ = [
        ("rows", c_int32), ("cols", c_int32), ("capacity", c_int64),
        ("row_ptr", c_void_p), ("col_idx", c_void_p), ("val", c_void_p),
        ("t_row_ptr", c_void_p), ("t_col_idx", c_void_p), ("t_val", c_void_p),
        ("t_pos", c_void_p),
    ]


class CsrtError(RuntimeError):
    pass


_LIB = None

_SIGS = {
    "csrt_workspace_bytes": [c_int32, c_int32, c_int32, POINTER(c_size_t)],
    "csrt_workspace_init": [c_void_p, c_size_t, c_void_p],
    "csrt_get_status": [c_void_p, POINTER(c_int32), POINTER(c_int64), c_void_p],
    "csrt_clear_status": [c_void_p, c_void_p],
    "csrt_validate_csr": [POINTER(csrt_csr), c_void_p, c_size_t, c_void_p],
    "csrt_get_invalid_row": [c_void_p, POINTER(c_int64), c_void_p],
    "csr_from_dense": [c_void_p, c_int32, c_int32, POINTER(csrt_csr), c_void_p, c_size_t, c_void_p],
    "csr_transpose": [POINTER(csrt_csr), c_void_p, c_size_t, c_void_p],
    "spmm_fwd": [POINTER(csrt_csr), c_void_p, c_int32, c_void_p, c_void_p, c_size_t, c_void_p],
    "spmm_bwd_t": [POINTER(csrt_csr), c_void_p, c_int32, c_void_p, c_void_p, c_size_t, c_void_p],
    "spmm_fwd_bias_act": [POINTER(csrt_csr), c_void_p, c_int32, c_void_p, c_int32, c_void_p, c_void_p, c_size_t,
                          c_void_p],
    "spmm_bwd_t_relu": [POINTER(csrt_csr), c_void_p, c_int32, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p],
    "spmm_fwd_noalloc": [POINTER(csrt_csr), c_void_p, c_int32, c_void_p, c_void_p],
    "spmm_fwd_noalloc_status": [POINTER(c_int32), c_int32, c_void_p],
    "weight_grad_dense": [c_void_p, c_void_p, c_int32, c_int32, c_int32, c_void_p, c_int32, c_void_p,
                          c_size_t, c_void_p],
    "weight_grad_sddmm": [POINTER(csrt_csr), c_void_p, c_void_p, c_int32, c_void_p, c_void_p, c_size_t,
                          c_void_p],
    "prox_update_compact": [POINTER(csrt_csr), c_void_p, c_float, c_float, POINTER(csrt_csr), c_void_p,
                            c_size_t, c_void_p],
    "debias_update": [POINTER(csrt_csr), c_void_p, c_float, c_void_p],
    "prox_rmsprop_update_compact": [POINTER(csrt_csr), c_void_p, c_void_p, c_float, c_float, c_float, c_float,
                                    POINTER(csrt_csr), c_void_p, c_size_t, c_void_p],
    "prox_adam_update_compact": [POINTER(csrt_csr), c_void_p, c_void_p, c_void_p, c_int32, c_float, c_float,
                                 c_float, c_float, c_float, POINTER(csrt_csr), c_void_p, c_size_t, c_void_p],
    "weight_grad_prox_update": [POINTER(csrt_csr), c_void_p, c_void_p, c_int32, c_float, c_float, c_int32, c_void_p,
                                POINTER(csrt_csr), c_void_p, c_size_t, c_void_p],
    "csrt_bias_act_fwd": [c_void_p, c_void_p, c_int32, c_int32, c_int32, c_void_p],
    "csrt_relu_bwd": [c_void_p, c_void_p, c_int64, c_void_p],
    "csrt_bias_grad_sgd": [c_void_p, c_int32, c_int32, c_void_p, c_float, c_void_p, c_void_p],
    "csrt_softmax_xent": [c_void_p, c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p],
    "csrt_im2col": [c_void_p, c_int32, c_int32, c_int32, c_int32, c_int32, c_void_p, c_void_p],
    "csrt_col2im": [c_void_p, c_int32, c_int32, c_int32, c_int32, c_int32, c_void_p, c_void_p],
    "csrt_check_bounded_waits": [c_void_p, c_size_t, c_void_p],
    "csrt_fma_peak_run": [c_void_p, c_int32, c_int32, ctypes.POINTER(ctypes.c_double), c_void_p],
    "csrt_conv2d_sparse_fwd": [POINTER(csrt_csr), c_void_p, c_int32, c_int32, c_int32, c_int32, c_int32, c_void_p,
                               c_int32, c_void_p, c_void_p],
    "csrt_maxpool2_fwd": [c_void_p, c_int32, c_int32, c_int32, c_int32, c_void_p, c_void_p, c_void_p],
    "csrt_maxpool2_bwd": [c_void_p, c_void_p, c_int32, c_int32, c_int32, c_int32, c_void_p, c_void_p],
    "csrt_flatten": [c_void_p, c_int32, c_int32, c_int32, c_void_p, c_void_p],
    "csrt_unflatten": [c_void_p, c_int32, c_int32, c_int32, c_void_p, c_void_p],
}


def lib():
    """Load libcsrtrain.so once; raise if it has not been built."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise CsrtError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, args in _SIGS.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = c_int32
        L.csrt_last_error.argtypes = []
        L.csrt_last_error.restype = ctypes.c_char_p
        L.csrt_launch_count.argtypes = [c_int32]
        L.csrt_launch_count.restype = c_int64
        _LIB = L
    return _LIB


def exported_symbols():
    """The entry points this binding expects the library to export."""
    return sorted(list(_SIGS) + ["csrt_last_error", "csrt_launch_count"])


def _check(rc: int, what: str):
    if rc != CSRT_OK:
        msg = lib().csrt_last_error().decode(errors="replace")
        raise CsrtError(f"{what} failed with code {rc}: {msg}")


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return c_void_p(stream.cuda_stream)


def _ptr(t):
    return None if t is None else c_void_p(t.data_ptr())


def _f32(t, name, numel=None):
    if t.dtype != torch.float32 or not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous float32 CUDA tensor")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} has {t.numel()} elements, needs {numel}")
    return t


def launch_count(reset: bool = False) -> int:
    return int(lib().csrt_launch_count(1 if reset else 0))


# ---------------------------------------------------------------------------
# Owned device objects
# ---------------------------------------------------------------------------

class CSR:
    """A device CSR matrix (caller-owned torch buffers) with optional
    transposed arrays, mirroring ``csrt_csr``."""

    def __init__(self, rows: int, cols: int, capacity: int | None = None, transposed: bool = True,
                 device="cuda"):
        self.rows, self.cols = int(rows), int(cols)
        self.capacity = int(rows * cols if capacity is None else capacity)
        cap = max(self.capacity, 1)
        i32 = dict(dtype=torch.int32, device=device)
        self.row_ptr = torch.zeros(self.rows + 1, **i32)
        self.col_idx = torch.zeros(cap, **i32)
        self.val = torch.zeros(cap, dtype=torch.float32, device=device)
        self.transposed = transposed
        if transposed:
            self.t_row_ptr = torch.zeros(self.cols + 1, **i32)
            self.t_col_idx = torch.zeros(cap, **i32)
            self.t_val = torch.zeros(cap, dtype=torch.float32, device=device)
            self.t_pos = torch.zeros(cap, **i32)
        else:
            self.t_row_ptr = self.t_col_idx = self.t_val = self.t_pos = None
        self._s = csrt_csr(self.rows, self.cols, self.capacity, _ptr(self.row_ptr), _ptr(self.col_idx),
                           _ptr(self.val), _ptr(self.t_row_ptr), _ptr(self.t_col_idx), _ptr(self.t_val),
                           _ptr(self.t_pos))

    @property
    def struct(self):
        return ctypes.byref(self._s)

    def nnz(self) -> int:
        return int(self.row_ptr[self.rows].item())

    def copy_from(self, other: "CSR"):
        """Device-to-device copy of another CSR of the same shape (nnz entries)."""
        self.row_ptr.copy_(other.row_ptr)
        n = other.nnz()
        self.col_idx[:n].copy_(other.col_idx[:n])
        self.val[:n].copy_(other.val[:n])
        if self.transposed and other.transposed:
            self.t_row_ptr.copy_(other.t_row_ptr)
            self.t_col_idx[:n].copy_(other.t_col_idx[:n])
            self.t_val[:n].copy_(other.t_val[:n])
            self.t_pos[:n].copy_(other.t_pos[:n])

    def to_host(self):
        """(row_ptr, col_idx, val) as numpy arrays trimmed to nnz, and the
        transposed arrays (or None)."""
        n = self.nnz()
        main = (self.row_ptr.cpu().numpy(), self.col_idx[:n].cpu().numpy(), self.val[:n].cpu().numpy())
        if not self.transposed:
            return main, None
        t = (self.t_row_ptr.cpu().numpy(), self.t_col_idx[:n].cpu().numpy(), self.t_val[:n].cpu().numpy(),
             self.t_pos[:n].cpu().numpy())
        return main, t


class Workspace:
    """Device scratch + status word (csrt_workspace_bytes / csrt_workspace_init)."""

    def __init__(self, rows: int, cols: int, max_n: int, device="cuda", stream=None):
        nbytes = c_size_t(0)
        _check(lib().csrt_workspace_bytes(int(rows), int(cols), int(max_n), ctypes.byref(nbytes)),
               "csrt_workspace_bytes")
        self.nbytes = int(nbytes.value)
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        _check(lib().csrt_workspace_init(_ptr(self.buf), self.nbytes, _stream(stream)), "csrt_workspace_init")

    @property
    def ptr(self):
        return _ptr(self.buf)

    def status(self, stream=None):
        flags, req = c_int32(0), c_int64(0)
        _check(lib().csrt_get_status(self.ptr, ctypes.byref(flags), ctypes.byref(req), _stream(stream)),
               "csrt_get_status")
        return int(flags.value), int(req.value)

    def clear_status(self, stream=None):
        _check(lib().csrt_clear_status(self.ptr, _stream(stream)), "csrt_clear_status")


# ---------------------------------------------------------------------------
# The training-step calls
# ---------------------------------------------------------------------------

def csr_from_dense(dense: torch.Tensor, out: CSR, ws: Workspace, stream=None):
    _f32(dense, "dense", out.rows * out.cols)
    _check(lib().csr_from_dense(_ptr(dense), out.rows, out.cols, out.struct, ws.ptr, ws.nbytes, _stream(stream)),
           "csr_from_dense")


def validate_csr(w: CSR, ws: Workspace, stream=None):
    """Structural check of w (and its transposed copy). Returns the first row
    with a broken invariant (see csrt_get_invalid_row), or None. Synchronises;
    leaves CSRT_DEV_INVALID set in the status word when it finds one."""
    _check(lib().csrt_validate_csr(w.struct, ws.ptr, ws.nbytes, _stream(stream)), "csrt_validate_csr")
    row = c_int64(0)
    _check(lib().csrt_get_invalid_row(ws.ptr, ctypes.byref(row), _stream(stream)), "csrt_get_invalid_row")
    return None if row.value < 0 else int(row.value)


def csr_transpose(w: CSR, ws: Workspace, stream=None):
    _check(lib().csr_transpose(w.struct, ws.ptr, ws.nbytes, _stream(stream)), "csr_transpose")


def spmm_fwd(w: CSR, x: torch.Tensor, y: torch.Tensor, ws: Workspace, stream=None):
    n = x.shape[1] if x.dim() == 2 else x.numel() // max(w.cols, 1)
    _f32(x, "X", w.cols * n)
    _f32(y, "Y", w.rows * n)
    _check(lib().spmm_fwd(w.struct, _ptr(x), n, _ptr(y), ws.ptr, ws.nbytes, _stream(stream)), "spmm_fwd")


def spmm_bwd_t(w: CSR, dy: torch.Tensor, dx: torch.Tensor, ws: Workspace, stream=None):
    n = dy.shape[1] if dy.dim() == 2 else dy.numel() // max(w.rows, 1)
    _f32(dy, "dY", w.rows * n)
    _f32(dx, "dX", w.cols * n)
    _check(lib().spmm_bwd_t(w.struct, _ptr(dy), n, _ptr(dx), ws.ptr, ws.nbytes, _stream(stream)), "spmm_bwd_t")


def spmm_fwd_bias_act(w: CSR, x: torch.Tensor, bias, relu: bool, y: torch.Tensor, ws: Workspace, stream=None):
    n = x.shape[1] if x.dim() == 2 else x.numel() // max(w.cols, 1)
    _f32(x, "X", w.cols * n)
    _f32(y, "Y", w.rows * n)
    if bias is not None:
        _f32(bias, "bias", w.rows)
    _check(lib().spmm_fwd_bias_act(w.struct, _ptr(x), n, _ptr(bias), 1 if relu else 0, _ptr(y), ws.ptr, ws.nbytes,
                                   _stream(stream)), "spmm_fwd_bias_act")


def spmm_bwd_t_relu(w: CSR, dy: torch.Tensor, y_below: torch.Tensor, dx: torch.Tensor, ws: Workspace, stream=None):
    n = dy.shape[1] if dy.dim() == 2 else dy.numel() // max(w.rows, 1)
    _f32(dy, "dY", w.rows * n)
    _f32(dx, "dX", w.cols * n)
    _f32(y_below, "y_below", w.cols * n)
    _check(lib().spmm_bwd_t_relu(w.struct, _ptr(dy), n, _ptr(y_below), _ptr(dx), ws.ptr, ws.nbytes, _stream(stream)),
           "spmm_bwd_t_relu")


def spmm_fwd_noalloc(w: CSR, x: torch.Tensor, y: torch.Tensor, stream=None):
    """spmm_fwd without a workspace (the library's own fixed device scratch)."""
    n = x.shape[1] if x.dim() == 2 else x.numel() // max(w.cols, 1)
    _f32(x, "X", w.cols * n)
    _f32(y, "Y", w.rows * n)
    _check(lib().spmm_fwd_noalloc(w.struct, _ptr(x), n, _ptr(y), _stream(stream)), "spmm_fwd_noalloc")


def weight_grad_dense(dy: torch.Tensor, x: torch.Tensor, g: torch.Tensor, ws: Workspace,
                      precision: int = CSRT_PREC_FP32, stream=None):
    m, n = dy.shape
    k = x.shape[0]
    if x.shape[1] != n:
        raise ValueError("dY and X must have the same number of columns")
    _f32(dy, "dY")
    _f32(x, "X")
    _f32(g, "G", m * k)
    _check(lib().weight_grad_dense(_ptr(dy), _ptr(x), m, k, n, _ptr(g), int(precision), ws.ptr, ws.nbytes,
                                   _stream(stream)), "weight_grad_dense")


def weight_grad_sddmm(w: CSR, dy: torch.Tensor, x: torch.Tensor, g: torch.Tensor, ws: Workspace, stream=None):
    n = dy.shape[1]
    _f32(dy, "dY", w.rows * n)
    _f32(x, "X", w.cols * n)
    _f32(g, "g", 1)
    _check(lib().weight_grad_sddmm(w.struct, _ptr(dy), _ptr(x), n, _ptr(g), ws.ptr, ws.nbytes, _stream(stream)),
           "weight_grad_sddmm")


def prox_update_compact(w_in: CSR, g: torch.Tensor, eta: float, lam: float, w_out: CSR, ws: Workspace,
                        stream=None):
    _f32(g, "G", w_in.rows * w_in.cols)
    _check(lib().prox_update_compact(w_in.struct, _ptr(g), float(eta), float(lam), w_out.struct, ws.ptr,
                                     ws.nbytes, _stream(stream)), "prox_update_compact")


def prox_rmsprop_update_compact(w_in: CSR, g: torch.Tensor, v: torch.Tensor, eta: float, lam: float, beta: float,
                                eps: float, w_out: CSR, ws: Workspace, stream=None):
    """One Prox-RMSProp step (Algorithm 1); v (M x K) is updated in place."""
    _f32(g, "G", w_in.rows * w_in.cols)
    _f32(v, "v", w_in.rows * w_in.cols)
    _check(lib().prox_rmsprop_update_compact(w_in.struct, _ptr(g), _ptr(v), float(eta), float(lam), float(beta),
                                             float(eps), w_out.struct, ws.ptr, ws.nbytes, _stream(stream)),
           "prox_rmsprop_update_compact")


def prox_adam_update_compact(w_in: CSR, g: torch.Tensor, m: torch.Tensor, v: torch.Tensor, t: int, eta: float,
                             lam: float, beta1: float, beta2: float, eps: float, w_out: CSR, ws: Workspace,
                             stream=None):
    """Step t >= 1 of Prox-ADAM (Algorithm 2); m and v (M x K) are updated in place."""
    _f32(g, "G", w_in.rows * w_in.cols)
    _f32(m, "m", w_in.rows * w_in.cols)
    _f32(v, "v", w_in.rows * w_in.cols)
    _check(lib().prox_adam_update_compact(w_in.struct, _ptr(g), _ptr(m), _ptr(v), int(t), float(eta), float(lam),
                                          float(beta1), float(beta2), float(eps), w_out.struct, ws.ptr, ws.nbytes,
                                          _stream(stream)), "prox_adam_update_compact")


def weight_grad_prox_update(w_in: CSR, dy: torch.Tensor, x: torch.Tensor, eta: float, lam: float, w_out: CSR,
                            ws: Workspace, precision: int = CSRT_PREC_TF32, g_scratch=None, stream=None):
    n = dy.shape[1]
    _f32(dy, "dY", w_in.rows * n)
    _f32(x, "X", w_in.cols * n)
    if g_scratch is not None:
        _f32(g_scratch, "g_scratch", w_in.rows * w_in.cols)
    _check(lib().weight_grad_prox_update(w_in.struct, _ptr(dy), _ptr(x), n, float(eta), float(lam), int(precision),
                                         _ptr(g_scratch), w_out.struct, ws.ptr, ws.nbytes, _stream(stream)),
           "weight_grad_prox_update")


def debias_update(w: CSR, g: torch.Tensor, eta: float, stream=None):
    _f32(g, "g", 1)
    _check(lib().debias_update(w.struct, _ptr(g), float(eta), _stream(stream)), "debias_update")


# ---------------------------------------------------------------------------
# Glue
# ---------------------------------------------------------------------------

def bias_act_fwd(y, bias, relu: bool, stream=None):
    m, n = y.shape
    _f32(y, "y")
    _check(lib().csrt_bias_act_fwd(_ptr(y), _ptr(bias), m, n, 1 if relu else 0, _stream(stream)),
           "csrt_bias_act_fwd")


def relu_bwd(dy, y, stream=None):
    _f32(dy, "dy")
    _f32(y, "y", dy.numel())
    _check(lib().csrt_relu_bwd(_ptr(dy), _ptr(y), dy.numel(), _stream(stream)), "csrt_relu_bwd")


def bias_grad_sgd(dy, bias, eta: float, gb=None, stream=None):
    m, n = dy.shape
    _f32(dy, "dy")
    _check(lib().csrt_bias_grad_sgd(_ptr(dy), m, n, _ptr(bias), float(eta), _ptr(gb), _stream(stream)),
           "csrt_bias_grad_sgd")


def softmax_xent(z, labels, dz, loss, stream=None):
    c, n = z.shape
    _f32(z, "z")
    _f32(dz, "dz", c * n)
    _f32(loss, "loss", n + 1)
    if labels.dtype != torch.int32 or not labels.is_cuda:
        raise ValueError("labels must be int32 CUDA")
    _check(lib().csrt_softmax_xent(_ptr(z), _ptr(labels), c, n, _ptr(dz), _ptr(loss), _stream(stream)),
           "csrt_softmax_xent")


def im2col(x, c, b, h, w, k, cols, stream=None):
    _check(lib().csrt_im2col(_ptr(_f32(x, "x")), c, b, h, w, k, _ptr(_f32(cols, "cols")), _stream(stream)),
           "csrt_im2col")


def check_bounded_waits(ws: Workspace, stream=None):
    """Run the library's bounded waits against events that never happen; they
    must give up and set CSRT_DEV_TIMEOUT (read it with ws.status())."""
    _check(lib().csrt_check_bounded_waits(ws.ptr, ws.nbytes, _stream(stream)), "csrt_check_bounded_waits")


def fma_peak_tflops(reps: int = 5) -> float:
    """Measured FP32 FMA throughput of the current GPU (TFLOP/s): the median of
    `reps` timed runs of the library's FMA probe (two waves of blocks per SM,
    after a warm-up run), timed with CUDA events on the current stream."""
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    blocks, iters = 4 * sms, 1 << 15
    out = torch.empty(blocks * 512, dtype=torch.float32, device="cuda")
    flops = ctypes.c_double(0.0)
    s = torch.cuda.current_stream()

    def run():
        _check(lib().csrt_fma_peak_run(_ptr(out), blocks, iters, ctypes.byref(flops), _stream(s)),
               "csrt_fma_peak_run")

    run()
    times = []
    for _ in range(reps):
        st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        st.record(s)
        run()
        en.record(s)
        en.synchronize()
        times.append(st.elapsed_time(en) / 1e3)
    times.sort()
    return flops.value / times[len(times) // 2] / 1e12


def conv2d_sparse_fwd(w: CSR, x, c, b, h, wd, k, bias, relu, y, stream=None):
    """Convolution with CSR filters read straight from the input (no unfolded matrix)."""
    _f32(x, "x", c * b * h * wd)
    _f32(y, "y", w.rows * b * (h - k + 1) * (wd - k + 1))
    bp = _ptr(_f32(bias, "bias", w.rows)) if bias is not None else None
    _check(lib().csrt_conv2d_sparse_fwd(w.struct, _ptr(x), c, b, h, wd, k, bp, int(bool(relu)), _ptr(y),
                                        _stream(stream)), "csrt_conv2d_sparse_fwd")


def col2im(dcols, c, b, h, w, k, dx, stream=None):
    _check(lib().csrt_col2im(_ptr(_f32(dcols, "dcols")), c, b, h, w, k, _ptr(_f32(dx, "dx")), _stream(stream)),
           "csrt_col2im")


def maxpool2_fwd(x, c, b, h, w, y, idx, stream=None):
    _check(lib().csrt_maxpool2_fwd(_ptr(_f32(x, "x")), c, b, h, w, _ptr(_f32(y, "y")), _ptr(idx), _stream(stream)),
           "csrt_maxpool2_fwd")


def maxpool2_bwd(dy, idx, c, b, h, w, dx, stream=None):
    _check(lib().csrt_maxpool2_bwd(_ptr(_f32(dy, "dy")), _ptr(idx), c, b, h, w, _ptr(_f32(dx, "dx")),
                                   _stream(stream)), "csrt_maxpool2_bwd")


def flatten(x, c, b, hw, xf, stream=None):
    _check(lib().csrt_flatten(_ptr(_f32(x, "x")), c, b, hw, _ptr(_f32(xf, "xf")), _stream(stream)), "csrt_flatten")


def unflatten(xf, c, b, hw, x, stream=None):
    _check(lib().csrt_unflatten(_ptr(_f32(xf, "xf")), c, b, hw, _ptr(_f32(x, "x")), _stream(stream)),
           "csrt_unflatten")
