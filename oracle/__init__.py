"""CPU oracle for the TreeGraft verify-and-grow step.

Test infrastructure only: imported by tests/, the package smoke check and the
benchmark's CPU-baseline leg, never by the library itself.
"""
from .treegraft_oracle import *  # noqa: F401,F403
