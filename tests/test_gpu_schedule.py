"""The two Newton-Schulz schedules (one launch per product, or one persistent
launch with per-matrix dependency counters) compute every tile with the same
arithmetic, so every result must be bitwise identical; the persistent one is
also checked against the oracle directly (it is the default schedule, which
every other GPU parity test runs)."""
import numpy as np
import pytest

import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import Run

pytestmark = pytest.mark.gpu

RAGGED = ((200, 328), (392, 136), (8, 8), (136, 1000), (520, 520), (64, 2056), (1032, 264),
          (256, 512))
# ten NS frames: two persistent launches (at most eight classes each)
TEN_CLASSES = tuple((64 * (i + 1), 512) for i in range(8)) + ((520, 8), (16, 16))


def run_both(wl, steps, w_dtypes=None, ns_coeffs=None):
    import torch
    kw = {} if ns_coeffs is None else {"ns_coeffs": ns_coeffs}
    out = []
    for sched in (malt.MALT_NS_PHASED, malt.MALT_NS_PERSISTENT):
        run = Run(wl, check=[], w_dtypes=w_dtypes, **kw)
        run.opt.set_ns_schedule(sched)
        for _ in range(steps):
            run.step(oracle=False)
        assert run.status() == malt.MALT_OK
        torch.cuda.synchronize()
        res = [run.host(t) for t in run.W + run.M + run.l + run.r]
        res += [run.host(run.opt.direction(i)) for i in range(len(wl.shapes))]
        res.append(np.asarray(run.opt.debug_scalars()))
        out.append(res)
        run.close()
    for a, b in zip(*out):
        assert np.array_equal(a, b)


@pytest.mark.parametrize("variant", ["malt", "malter"])
def test_ragged_bitwise(variant):
    wl = inputs.Workload("sched", 50, RAGGED, "f32", 1.5, 0.02, variant, 3)
    run_both(wl, 3, w_dtypes=["f32", "bf16"] * 4)


@pytest.mark.parametrize("ns_steps", [1, 8])
def test_iteration_counts_bitwise(ns_steps):
    wl = inputs.Workload("schedk", 51, RAGGED[:5], "f32", 1.5, 0.02, "malt", 2, ns_steps=ns_steps)
    run_both(wl, 2)


def test_two_launch_groups_bitwise():
    wl = inputs.Workload("sched10", 52, TEN_CLASSES, "f32", 1.0, 0.02, "malt", 2)
    run_both(wl, 2)


def test_gpt2_large_layers_bitwise():
    wl = inputs.first_layers(inputs.WORKLOADS["gpt2_large"], 2)
    run_both(wl, 2)


def test_persistent_against_oracle_two_groups():
    wl = inputs.Workload("sched10o", 53, TEN_CLASSES, "f32", 1.0, 0.02, "malter", 2)
    run = Run(wl)
    run.opt.set_ns_schedule(malt.MALT_NS_PERSISTENT)
    for s in range(wl.steps):
        run.step()
        assert run.status() == malt.MALT_OK
        for i in range(len(wl.shapes)):
            run.assert_close(i, f"step {s}")
    run.close()


def test_unknown_schedule_rejected():
    wl = inputs.Workload("schedbad", 54, ((256, 512),), "f32", 1.0, 0.02, "malt", 1)
    run = Run(wl, check=[])
    with pytest.raises(malt.MaltError):
        run.opt.set_ns_schedule(7)
    run.close()
