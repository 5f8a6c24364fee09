"""Reference oracle for the SLORR regularizer hot path (test infrastructure only).

This package is a plain, slow, fp64 CPU restatement of what the regularizer
computes, written from the paper (SLORR, arXiv 2607.08754):

* ``schedule``       -- the Polar Express coefficient schedule (greedy minimax
  odd quintics, Sec. 3 "Computing the polar factor", App. C.1) and the scalar
  map it induces on singular values.
* ``slorr``          -- the per-matrix forward value and gradient of
  SLORR-Hoyer and SLORR-Nuc (Sec. 3 problem statement and Eq. 1, Listing 1,
  Alg. 2), the exact SVD-based quantities, and the FLOP model of Sec. 3
  "Computational cost".
* ``descent``        -- the regularizer-only descent step (last line of Alg. 1
  with no task update; the setting of Props. 2 and 3) and the retained-energy
  metric E(P) and rank P* of App. D.4.
* ``svd_jacobi``     -- an independent one-sided Jacobi SVD used only as a
  brute-force second opinion on tiny inputs.

It is test infrastructure: only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import it.  The CUDA path never
imports it, and it imports nothing from the CUDA path.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, invariants, brute force or the paper's bounds, except
the fidelity of the *default* schedule options (cushion and safety factor) to
the cited Polar Express work, which the paper does not print: that part is
"parity unpinned" (the schedule is pinned to its own definition, not to the
cited authors' constants).
"""

from .schedule import (  # noqa: F401
    minimax_odd_quintic,
    cushion_ratio,
    pe_schedule,
    pe_coefficients,
    pe_scalar_map,
    paper_delta,
    achieved_error,
)
from .slorr import (  # noqa: F401
    frobenius,
    polar_express,
    polar_express_steps,
    reg_forward_backward,
    reg_single,
    exact_values,
    exact_grad,
    pe_flops,
    weight_set_flops,
)
from .descent import (  # noqa: F401
    descent_step,
    descent_trajectory,
    singular_values,
    hoyer_tau,
    energy,
    energy_rank,
)
