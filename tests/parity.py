"""Comparison rules for GPU results against the CPU oracle.

Float32 results pass if |gpu - ref| <= atol + rtol*|ref| (rtol 1e-4, atol
1e-6; rtol 1e-3 for TF32 tensor-core products). An entry that misses this
(cancellation: |ref| much smaller than the terms it sums) must still meet the
worst-case summation bound |gpu - ref| <= gamma_n * S + unit*|ref|, where
S = sum |terms| (computed by the oracle on |W| and |X|; ``bound`` may be a
callable returning S, evaluated only when some entry misses the first test),
n the number of terms, gamma_n = n*u / (1 - n*u) with u = 2^-24, and for TF32 operands an
extra 2 * 2^-10 * S for the truncation of both factors. Integer arrays and
sparsity patterns are compared bit for bit.
"""

from __future__ import annotations

import numpy as np

U32 = 2.0 ** -24
TF32_OPERAND = 2.0 ** -10


def gamma(n, u=U32):
    n = np.asarray(n, dtype=np.float64)
    return n * u / (1.0 - n * u)


def assert_close(gpu, ref, bound=None, n_terms=None, rtol=1e-4, atol=1e-6, tf32=False, what=""):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    if gpu.size == 0:
        return 0
    err = np.abs(gpu - ref)
    ok = err <= atol + rtol * np.abs(ref)
    if ok.all():
        return 0
    bad = ~ok
    if bound is None or n_terms is None:
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{what}: {bad.sum()} entries off, e.g. {[(tuple(i), gpu[tuple(i)], ref[tuple(i)]) for i in idx]}")
    if callable(bound):
        bound = bound()
    s = np.broadcast_to(np.asarray(bound, dtype=np.float64), ref.shape)
    nt = np.broadcast_to(np.asarray(n_terms, dtype=np.float64), ref.shape)
    lim = gamma(nt + 1) * s + U32 * np.abs(ref) + 1e-30
    if tf32:
        lim = lim + 2 * TF32_OPERAND * s
    ok2 = err <= lim
    if not ok2[bad].all():
        idx = np.argwhere(bad & ~ok2)[:5]
        raise AssertionError(
            f"{what}: {int((bad & ~ok2).sum())} entries beyond the summation bound, e.g. "
            f"{[(tuple(i), gpu[tuple(i)], ref[tuple(i)], lim[tuple(i)]) for i in idx]}")
    return int(bad.sum())


def csr_dense(row_ptr, col_idx, val, rows, cols):
    d = np.zeros((rows, cols), dtype=np.float32)
    r = np.repeat(np.arange(rows), np.diff(np.asarray(row_ptr, dtype=np.int64)))
    d[r, col_idx] = val
    return d
