"""Seeded synthetic workloads shared by the tests, the smoke check and the
benchmark.  Holds random draws and shapes only, none of the method's
arithmetic."""
from .synth import *  # noqa: F401,F403
