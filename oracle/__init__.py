"""CPU oracle (test infrastructure only): imported by tests/, smoke() and bench.py's cpu_baseline leg."""
from .cast_oracle import *  # noqa: F401,F403
