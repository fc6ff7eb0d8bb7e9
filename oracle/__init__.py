"""CPU oracle for the UniQuan_F weight quantizer -- TEST INFRASTRUCTURE ONLY.

This package is a plain, slow, single-threaded numpy restatement of what the
UniQuan_F quantizer computes (arXiv 2506.03781, "Unifying Uniform and
Binary-coding Quantization for Accurate Compression of Large Language
Models").  It exists to check the CUDA library, never to stand in for it:

* only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
  ``--impl reference`` legs of ``bench.py`` may import or call it;
* it imports nothing from the CUDA package and the CUDA package imports
  nothing from here; the seeded input generators
  (``paper_2506_03781_gb300.synth``) are the only code both sides use, and
  they hold none of the method's arithmetic.

Precision policy (the paper fixes none):

* every value that DECIDES an integer -- the transformed weight x, the BCQ
  level values, the distances |x - level|, the gradient-filter test
  |x - level| <= tau -- is computed in IEEE fp32 with one stated operation
  order, because the kernels take the same decisions in fp32;
* every gradient value and every reduction is computed in fp64.

Every function is pinned by a ``-m "not gpu"`` test against something other
than itself (brute force, closed forms, invariants, finite differences,
library routines); see ``tests/test_oracle_*.py``.
"""

from .uniquan import *  # noqa: F401,F403
from .uniquan import __all__  # noqa: F401
