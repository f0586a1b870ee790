"""Plain CPU oracle for the Sigma-Delta-quantized (SDQ) linear layer.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
link this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code, tables or constants with the CUDA library in
``paper_2510_03275_gb300/``; the two meet only through the seeded inputs made
by ``paper_2510_03275_gb300.workloads``.

See ``oracle/sdq_oracle.py`` for the definitions and their citations.
"""
from .sdq_oracle import *  # noqa: F401,F403
