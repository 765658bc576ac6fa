"""fp64 CPU oracle of the LoCA hot path.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / reference arm of ``bench.py``, never by the CUDA library or its
Python binding.  See ``oracle/loca_oracle.py`` for the functions and their citations.
"""

from .loca_oracle import *  # noqa: F401,F403
from .loca_oracle import __all__  # noqa: F401
