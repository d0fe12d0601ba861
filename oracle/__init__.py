"""fp64 CPU oracle of the SBD block step -- test infrastructure only.

Imported by tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg;
never by the product package."""
from .sbd_oracle import *  # noqa: F401,F403
