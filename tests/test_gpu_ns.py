"""The Newton-Schulz engine stage by stage.  With one iteration and the
coefficients (a, b, c) set to (1, 0, 0), (0, 1, 0) and (0, 0, 1), the output
is X0, A X0 = X0 X0^T X0 and A^2 X0, which exercises the prescale and the BX
epilogue alone, then the Gram and BX GEMMs, then all three GEMMs.  Compared
with the oracle's Newton-Schulz on the oracle's Mt."""
import numpy as np
import pytest

import oracle.malt_ref as ref
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import Run, rel

pytestmark = pytest.mark.gpu

SHAPES = ((128, 256), (256, 512), (200, 328), (392, 136), (8, 8), (520, 1544))


@pytest.mark.parametrize("coeffs", [(1.0, 0.0, 0.0), (0.0, 1.0, 0.0), (0.0, 0.0, 1.0),
                                    (3.4445, -4.7750, 2.0315)])
def test_one_iteration(coeffs):
    wl = inputs.Workload("ns1", 50, SHAPES, "f32", 1.0, 0.02, "malt", 1, ns_steps=1)
    run = Run(wl, ns_coeffs=coeffs)
    run.step()
    assert run.status() == 0
    for i, shape in enumerate(SHAPES):
        want = ref.newton_schulz(run.info[i]["Mt"], 1, coeffs)
        got = run.host(run.opt.direction(i))
        assert got.shape == want.shape
        e = rel(got, want)
        assert e < 1e-2, (coeffs, shape, e)
    run.close()


def test_five_iterations_direction():
    wl = inputs.Workload("ns5", 51, SHAPES, "f32", 1.5, 0.02, "malt", 1)
    run = Run(wl)
    run.step()
    assert run.status() == 0
    for i, shape in enumerate(SHAPES):
        e = rel(run.host(run.opt.direction(i)), run.info[i]["O"])
        assert e < 2e-2, (shape, e)
    run.close()
