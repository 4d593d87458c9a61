"""fp64 CPU oracle (test infrastructure only; see ``arckv_oracle``).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline and
reference legs of ``bench.py`` may import this package.  It shares no code
with the CUDA library.
"""
from .arckv_oracle import *  # noqa: F401,F403
from .arckv_oracle import __all__  # noqa: F401
