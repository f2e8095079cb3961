"""Separate optimizer states share nothing: two states stepped at the same time
on two streams give bitwise the results of stepping them one after the other.

A race on anything the library kept between states (a device-side scratch
buffer, a work table, a counter) would show up as a difference; determinism
within one state is covered by the parity tests."""
import numpy as np
import pytest

import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import Run

pytestmark = pytest.mark.gpu

SHAPES_A = ((200, 328), (392, 136), (520, 520), (1032, 264))
SHAPES_B = ((256, 512), (64, 2056), (136, 1000), (777, 301))


def _states():
    import torch
    wa = inputs.Workload("concA", 60, SHAPES_A, "f32", 1.5, 0.02, "malt", 3)
    wb = inputs.Workload("concB", 61, SHAPES_B, "f32", 1.5, 0.02, "malter", 3)
    a = Run(wa, check=[], w_dtypes=["bf16", "f32"] * 2)
    b = Run(wb, check=[], w_dtypes=["f32", "bf16"] * 2)
    a.opt.set_ns_schedule(malt.MALT_NS_PERSISTENT)
    b.opt.set_ns_schedule(malt.MALT_NS_PHASED)
    for run in (a, b):
        for i in range(len(run.wl.shapes)):
            run.G[i].copy_(torch.from_numpy(run.gradient(i, 0)))
    torch.cuda.synchronize()
    return a, b


def _results(run):
    out = [run.host(t) for t in run.W + run.M + run.l + run.r]
    out += [run.host(run.opt.direction(i)) for i in range(len(run.wl.shapes))]
    nu, t = run.opt.scalars()
    return out + [np.asarray(nu), np.asarray([t])]


def test_two_states_on_two_streams_match_sequential():
    import torch
    a, b = _states()
    for _ in range(3):
        a.opt.step(a.hp)
        b.opt.step(b.hp, malter=True)
    torch.cuda.synchronize()
    assert a.status() == malt.MALT_OK and b.status() == malt.MALT_OK
    want_a, want_b = _results(a), _results(b)
    a.close()
    b.close()

    a, b = _states()
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    sa.wait_stream(torch.cuda.current_stream())
    sb.wait_stream(torch.cuda.current_stream())
    for _ in range(3):
        a.opt.step(a.hp, stream=sa)
        b.opt.step(b.hp, malter=True, stream=sb)
    torch.cuda.synchronize()
    assert a.status() == malt.MALT_OK and b.status() == malt.MALT_OK
    for k, (x, y) in enumerate(zip(_results(a), want_a)):
        assert np.array_equal(x, y), ("state A", k)
    for k, (x, y) in enumerate(zip(_results(b), want_b)):
        assert np.array_equal(x, y), ("state B", k)
    a.close()
    b.close()
