"""fp64 CPU oracle for ResKV (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs may import this package.  It shares no code with the CUDA
library and imports nothing from it.
"""
from .reskv_oracle import *  # noqa: F401,F403
from .reskv_oracle import (OracleConfig, UnitCache, GATE_DYNAMIC, GATE_FIXED,  # noqa: F401
                           SCORE_OBS_POOL, SCORE_KEYNORM, SOFTMAX_SHARED, SOFTMAX_SEPARATE)
