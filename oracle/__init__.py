"""CPU oracle for the heterogeneous data-parallel SGD step (arXiv 2110.08941).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (the C-ABI library and its Python binding) never
imports, links or runs anything here, and this package imports nothing from
the product: the two share no code.  The only shared module is ``synth``, the
seeded input generator, which holds none of the method's arithmetic.

Plain, slow, obviously correct fp64 NumPy, written from the paper:

* ``oracle.partition`` - Section 4, Eq. 2 (compute power), Eq. 3 (predicted
  time) and Algorithm 1 (Dynamic Partitioning), with the integer-rounding
  reading stated in that module.
* ``oracle.mlp`` / ``oracle.cnn`` - Eq. 1 (per-worker mean loss f_m) and its
  gradient g^m by explicit back-propagation, for the MLP and CNN workloads.
* ``oracle.sgd`` - the synchronisation of Section 1 (g = (1/M) sum_m g^m), the
  compute-power weighting of Section 4.2 (Enhanced DP), and the update
  theta <- theta - eta * g of Section 1.

Pins (tests/test_oracle_*.py) tie each function to something other than
itself: worked partitions, closed-form invariants, brute force over tiny
cases, central finite differences, and torch.autograd / torch.optim.SGD in
fp64 as independent library routines.  No function here is "parity unpinned".
"""
from . import partition, mlp, cnn, sgd  # noqa: F401
