"""CPU oracle for the slice -> mix -> deslice coupling (test infrastructure).

This package is the independent, slow and plain reference that the CUDA
library is checked against.  Only tests/, __graft_entry__.smoke() and the
CPU-baseline leg of bench.py may import it.  The library never imports it,
shares no code with it, and has no CPU fallback to it.

  flashslice_oracle  fp64 numpy, materialised slice weights (the definition)
  bruteforce         scalar Python loops on tiny inputs (pins the former)

Pins: every function here is checked by tests/test_oracle_pins.py against
values fixed by the paper's definitions and by mathematics (a hand-derived
worked example in tests/golden/, closed forms, invariants, finite
differences, the scalar-loop restatement).  The mapping of each function to
its pins is in the module docstrings and the test file; no function is
"parity unpinned".
"""
from . import flashslice_oracle  # noqa: F401
from .flashslice_oracle import (  # noqa: F401
    DEFAULT_EPS, backward, deslice_bwd, deslice_fwd, forward, logits, mix, mix_bwd,
    slice_bwd, slice_finalize, slice_fwd, softmax_rows,
)
