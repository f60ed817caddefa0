"""CPU oracle of the RPD commit step (fp64).  Test infrastructure only: imported by
``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline and reference legs,
never by the library."""
from .rpd_oracle import *  # noqa: F401,F403
from .rpd_oracle import RULES, StepResult  # noqa: F401
