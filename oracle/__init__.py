"""Plain CPU oracle for Chameleon's format-adaptive quantized linear layer.

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this package.  The
product path (the CUDA library and its Python binding) never imports, calls or links it, and
this package imports nothing from the product path.

Every function follows one passage of the paper (arXiv 2609.33496, "Chameleon"), cited in its
docstring by section / equation / algorithm.  Arithmetic is numpy: float64 for values and error
sums, float32 exactly where the format definitions fix an fp32 scale or product.  Nothing is
blocked, fused or reordered beyond the definitions.

Modules
  formats   number-format grids and codecs (Sec. 3.2, App. A.11, ScaleZP of App. A.7)
  schedule  SNR(t), bucket index, kurtosis, routing rule (Eq. 1, Sec. 3.3-3.5, Alg. 1-3)
  select    per-channel weight-format selection (Sec. 3.4, Eq. weight-argmax)
  gemm      fp64 reference of the quantized linear and its error bound
  nf4       NormalFloat-4 level construction (cited at App. A.11)

Pins: every function is checked against something outside itself (closed forms, worked values,
library routines, brute force, planted mistakes).  The NF4 levels, for which the paper cites
QLoRA without printing a table, are checked against the table QLoRA publishes
(``tests/golden/``).
"""
from . import formats, schedule, select, gemm, nf4  # noqa: F401
