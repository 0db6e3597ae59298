"""Seeded synthetic workloads shared by the tests, the smoke check and the
benchmark.  Holds none of the method's arithmetic."""
from .generate import *  # noqa: F401,F403
