"""CPU oracles of the FL-GLM server block stack (test infrastructure only).

flglm_oracle.py: fp64 numpy (the pinned reference of every definition, also the GLM mask,
P-tuning prefix and client parts); flglm_oracle32.cpp (+ oracle32.py): the same server
block stack, fp32 C++17 with OpenMP and no BLAS, cross-checked against the fp64 one and
timed as the CPU baseline.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
``cpu_baseline`` and ``--impl reference`` legs may import this package.  The CUDA library
never does.
"""
from .flglm_oracle import *  # noqa: F401,F403
from .flglm_oracle import OracleServer, Packing, BlockShape  # noqa: F401
