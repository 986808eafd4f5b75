"""CPU oracle of the Reflective Verification verify step (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference legs may import this package.  It shares no code with the CUDA path.
"""
from .rv_oracle import *  # noqa: F401,F403
from . import rv_oracle  # noqa: F401
