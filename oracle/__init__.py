"""CPU oracle for the permutation-group Allreduce (Kolmakov & Zhang, arXiv 2004.09362).

TEST INFRASTRUCTURE, NOT PRODUCT CODE. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline / ``--impl reference`` legs of ``bench.py`` may import or run anything
under ``oracle/``. The library in ``paper_2004_09362_gb300/`` never imports it, and the
two share no code: the only common dependency is the seeded input generator module
``gar_inputs``, which holds none of the method's arithmetic.

See ``oracle/gar_oracle.py`` for what is computed and which passage of the paper each
function follows.  Parity status: every function here is pinned by ``-m "not gpu"``
tests (``tests/test_oracle_pins.py``); each docstring names its pins ("Pinned by:").
"""

from .gar_oracle import *  # noqa: F401,F403
