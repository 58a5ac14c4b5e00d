"""CPU oracle for layer dropout (stochastic depth) on a pre-norm decoder stack.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute anything in this package: only ``tests/``, ``__graft_entry__.smoke()``
and the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.
The CUDA library and this package share no code, headers, tables or helpers;
the only shared module is the seeded input generator
(``paper_2609_05275_gb300/synth.py``), which holds none of the method's
arithmetic.

Everything here is plain and slow on purpose: numpy in float64, one sequence
at a time, library matmuls as the only primitive.  Each function names the
passage of the paper (arXiv 2609.05275, "Don't Drop Dropout") it follows.

Modules
  schedule  -- per-layer drop rates p^{l,t}: distributions x time schedules
               (Dropout Distribution / Dropout Schedule sections), the drop
               threshold and the residual scale r_train = 1/rho.
  philox    -- Philox4x32-10 (Salmon et al., SC'11), the counter-based RNG
               that draws the Bernoulli masks.
  masks     -- the masks M^{l,t} in {0,1}^B (Eq. layer_dropout_train) at
               per-sequence or per-batch granularity, and the kept lists.
  stack     -- forward and hand-derived backward of the transformer form of
               layer dropout (Eq. transformer_layer_dropout_train).

Parity status: every function here is pinned by a ``-m "not gpu"`` test
(closed forms and printed numbers of the paper, published Philox
known-answer vectors, a torch library reference with autograd, finite
differences, brute force over masks).  None is "parity unpinned".
"""

from . import schedule, philox, masks, stack  # noqa: F401
