"""CPU oracle for the LionMuon optimizer step.  Test infrastructure only:
imported by tests/, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline
legs, never by the product package."""

from .lionmuon_oracle import *  # noqa: F401,F403
from .lionmuon_oracle import Config, NS_QUINTIC, NS_CUBIC  # noqa: F401
