"""fp64 CPU oracle of the FL-GLM server block stack (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s ``cpu_baseline`` and
``--impl reference`` legs may import this package.  The CUDA library never does.
"""
from .flglm_oracle import *  # noqa: F401,F403
from .flglm_oracle import OracleServer, Packing, BlockShape  # noqa: F401
