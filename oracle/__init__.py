"""fp64 CPU oracle for the partial-straggler gradient-coding hot path.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` (and its ``--impl reference`` arm) may import
or run anything in this package.  The CUDA library never imports it and the two
share no code; the only things both sides receive are the seeded inputs that
``workloads`` produces.

Pin status (what fixes each function other than itself; tests/test_oracle_pins.py):
  cyclic_order / ordering_matrix / q_metric  -- Sec. III row-sum optimum, column permutations
  completed_sets / support / copies          -- worked example, eqs. (3) and (8) (tests/golden)
  find_encoding_coeff / encoding_matrix      -- closed forms of Sec. II-B (under- and
                                                over-determined), QR projector, rank identity
  encode / decode                            -- exact recovery (Sec. II-A), l = 1 remark,
                                                baseline scheme (Sec. I)
  chunk_gradient(s) / point_losses           -- finite differences, one-shot full gradient
  coefficient_error / error_estimate         -- per-pattern rank identity vs eq. (7)
  gradient_mse                               -- l = 1 closed form, exact patterns
  sgd_step / full_loss                       -- finite differences of L = (1/N~) sum l
"""
from .gc_oracle import *  # noqa: F401,F403
from . import gc_oracle  # noqa: F401
