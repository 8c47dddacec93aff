"""fp64 CPU oracle for progressive approximate-LSTM inference.

TEST INFRASTRUCTURE ONLY.  Nothing in the product (the CUDA library and its
Python binding) may import, call or link anything in this package; only the
tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py``
use it.  It shares no code with the CUDA path: the only module both sides
import is ``workloads`` (seeded random draws, none of the method's
arithmetic).

Two parts, each written from the paper in its order and notation:

* :mod:`oracle.factors` -- the offline approximation of Sec. III: augmented
  gate matrix, rank-1 SVD of the residual, magnitude pruning of v, residual
  refinement (Eq. 1 and the residual definition that follows it).
* :mod:`oracle.recurrence` -- the LSTM recurrence of Sec. II / Fig. 2 with
  each gate's matrix-vector product replaced by the refinement sum of Eq. 1,
  including outputs at intermediate refinement depths (progressive
  inference, Sec. I / Fig. 1b).

Everything is float64 with plain loops; NumPy's SVD, sort and dot serve as
library steps.  Pins against the paper and the mathematics live in
``tests/test_oracle_*.py``.
"""
from .factors import (decompose_gate, decompose_gate_variant, decompose_layer, prune, prune_dense,  # noqa: F401
                      reconstruct, top_triplet)
from .recurrence import run_lstm, lstm_cell, refinement_sums, op_count  # noqa: F401
