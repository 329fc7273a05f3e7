"""CPU oracle of ADEPT's early-exit forward pass.

TEST INFRASTRUCTURE ONLY: imported by the test suite, the smoke check and the
benchmark's CPU-baseline leg, never by the library itself.
"""
from .adept_oracle import *  # noqa: F401,F403
