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


SCHEDULES = [malt.MALT_NS_PHASED, malt.MALT_NS_PERSISTENT, malt.MALT_NS_AUTO]


def run_both(wl, steps, w_dtypes=None, ns_coeffs=None, schedules=SCHEDULES, g_dtype="f32"):
    """The same steps under every schedule: all results bitwise equal."""
    import torch
    kw = {"g_dtype": g_dtype}
    if ns_coeffs is not None:
        kw["ns_coeffs"] = ns_coeffs
    out = []
    for sched in schedules:
        run = Run(wl, check=[], w_dtypes=w_dtypes, **kw)
        run.opt.set_ns_schedule(sched)
        for _ in range(steps):
            run.step(oracle=False)
        assert run.status() == malt.MALT_OK, (sched, run.opt.timeout_site())
        torch.cuda.synchronize()
        res = [run.host(t) for t in run.W + run.M + run.l + run.r]
        res += [run.host(run.opt.direction(i)) for i in range(len(wl.shapes))]
        res.append(np.asarray(run.opt.debug_scalars()))
        nu, t = run.opt.scalars()
        res += [np.asarray(nu), np.asarray([t])]
        out.append(res)
        run.close()
    for sched, res in zip(schedules[1:], out[1:]):
        for i, (a, b) in enumerate(zip(out[0], res)):
            assert np.array_equal(a, b), (sched, i)


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


@pytest.mark.parametrize("seed,variant,g_dtype", [(4, "malter", "f32"), (5, "malter", "f32"),
                                                  (6, "malt", "bf16"), (7, "muon", "f32"),
                                                  (8, "malter", "bf16")])
def test_seeded_random_shapes_bitwise(seed, variant, g_dtype):
    shapes = inputs.random_shapes(seed, 10)
    wl = inputs.Workload(f"schedrand{seed}", 60 + seed, shapes, "f32", 1.5, 0.02, variant, 3)
    run_both(wl, 3, w_dtypes=["f32", "bf16"] * 5, g_dtype=g_dtype)


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


@pytest.mark.parametrize("schedule", [malt.MALT_NS_PERSISTENT, malt.MALT_NS_PHASED])
def test_ns_steps_change_between_steps(schedule):
    """One state stepped with ns_steps 5, 3, 5, 3: the persistent launches
    claim the first k iterations' entries of the work table built at init,
    and every step matches the oracle run with the same sequence."""
    import dataclasses
    wl = inputs.Workload("kswitch", 39, ((256, 512), (392, 136), (520, 520)), "f32", 1.0, 0.02,
                         "malter", 4)
    run = Run(wl, w_dtypes=["f32", "bf16", "f32"])
    run.opt.set_ns_schedule(schedule)
    base_ref = run.hp_ref
    for s, k in enumerate((5, 3, 5, 3)):
        run.hp_ref = dataclasses.replace(base_ref, ns_steps=k)
        run.hp = malt.hparams(lr=wl.lr, ns_steps=k)
        run.step()
        assert run.status() == malt.MALT_OK, run.opt.timeout_site()
        for i in range(len(wl.shapes)):
            run.assert_close(i, f"step {s} k={k}")
    run.close()


def test_unknown_schedule_rejected():
    wl = inputs.Workload("schedbad", 54, ((256, 512),), "f32", 1.0, 0.02, "malt", 1)
    run = Run(wl, check=[])
    with pytest.raises(malt.MaltError):
        run.opt.set_ns_schedule(7)
    run.close()


def test_column_major_bx_order_bitwise_and_against_oracle():
    """A frame whose X is larger than 32 MiB (2056 x 8192, bf16: 33.7 MB) lists
    its B*X tiles column by column; with a ragged last tile row (2056 = 8 x 257)
    both schedules agree bitwise and the step matches the oracle."""
    wl = inputs.Workload("bxcol", 57, ((2056, 8192),), "bf16", 1.5, 0.02, "malt", 1)
    run_both(wl, 1, schedules=[malt.MALT_NS_PHASED, malt.MALT_NS_PERSISTENT])
    run = Run(wl)
    run.step()
    assert run.status() == malt.MALT_OK
    run.assert_close(0)
    run.close()


def test_unaligned_shapes_bitwise():
    """Padded matrices (rows or cols not multiples of 8) give bitwise the same
    results under every schedule."""
    shapes = inputs.random_shapes(23, 10, max_dim=517, multiple=1)
    wl = inputs.Workload("schedodd", 58, shapes, "f32", 1.5, 0.02, "malter", 2)
    run_both(wl, 2, w_dtypes=["f32", "bf16"] * 5, g_dtype="bf16")
