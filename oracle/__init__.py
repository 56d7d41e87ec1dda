"""fp64 CPU oracle (test infrastructure only: used by tests/, smoke() and bench.py's CPU legs)."""
from .ssd_oracle import *  # noqa: F401,F403
