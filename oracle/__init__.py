"""fp64 CPU oracles for the MALT / MALTER update (malt_ref) and for the AdamW
update of the non-matrix parameters in a whole-optimizer step (adamw_ref).
Test infrastructure only: imported by the test suite, the package smoke check
and the benchmark's CPU baseline leg, never by the library."""
from .malt_ref import *  # noqa: F401,F403
from .malt_ref import Hyper, State, malt_step_ref, run_steps  # noqa: F401
