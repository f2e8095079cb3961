"""fp64 CPU oracle for the MALT / MALTER update.  Test infrastructure only:
imported by the test suite, the package smoke check and the benchmark's CPU
baseline leg, never by the library."""
from .malt_ref import *  # noqa: F401,F403
from .malt_ref import Hyper, State, malt_step_ref, run_steps  # noqa: F401
