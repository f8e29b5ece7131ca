"""CPU oracle for the CSR-weight training step of Lee & Lee, "Compressed Learning
of Deep Neural Networks for OpenCL-Capable Embedded Systems" (arXiv 1905.07931).

This package is TEST INFRASTRUCTURE. It is a plain, slow, obviously correct
restatement of what the training step computes, written from the paper's
definitions (Sections 2.1-2.4 and 3.1-3.3). Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it. The CUDA library never calls it and shares no code with it.

Precision: every sum is accumulated in float64 and rounded to float32 once.
The proximal step is the exception: it follows fixed float32 rounding rules
(see ``prox_update_compact``) so that the sparsity pattern it produces is
bit-exact and can be compared bit for bit.

Parity status per function is stated in each docstring ("pinned by ..."). The
only unpinned quantity is a free-running multi-step trajectory (GPU and oracle
gradients differ in summation order, so patterns may diverge after the first
step); it is compared step by step with the oracle re-fed the GPU gradient.
"""

from .csr_oracle import *  # noqa: F401,F403
from .csr_oracle import __all__  # noqa: F401
