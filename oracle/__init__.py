"""Float64 CPU oracle for the ACRL hot path.

Test infrastructure only: imported by the test-suite, the smoke check and the
CPU-baseline leg of the benchmark, never by the library or its binding.
"""
from .acrl_oracle import *  # noqa: F401,F403
from .acrl_oracle import Params, ControllerState, StepResult  # noqa: F401
