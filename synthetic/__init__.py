"""Seeded synthetic inputs (no arithmetic of the method): shared by tests, bench and smoke."""
from . import generators, workloads  # noqa: F401
