"""Plain fp64 CPU oracle for the DP-SGD gradient step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code, header, table or helper with the CUDA library; it reads the same
stored input bits (fp32 or bf16 upcast exactly to fp64) and computes every
quantity from its plain definition.

Pinning status (what ties each function to something other than itself) is
listed in the header of :mod:`oracle.dp_oracle`.
"""

from .dp_oracle import *  # noqa: F401,F403
