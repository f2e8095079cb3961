"""The CPU model of the kernel's bf16 Newton-Schulz arithmetic (tests only),
against the fp64 oracle: without rounding it is the oracle's iteration (the
first iteration's 1/||Mt|| scaling and aI folded into B' change nothing in
exact arithmetic); with bf16 rounding its error on ordinary inputs is that of
bf16 operands, well inside the 2e-2 bar, and on a thin matrix with three
singular values it reaches the bar."""
import numpy as np

import oracle.malt_ref as ref
from tests.bf16_ns_model import newton_schulz_bf16


def _rel(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def test_without_rounding_it_is_the_oracle_iteration():
    rng = np.random.default_rng(81)
    for shape in ((48, 160), (160, 48), (64, 64)):
        X = rng.standard_normal(shape) * np.exp(rng.standard_normal(shape[1]))[None, :]
        for k, coeffs in ((5, ref.DEFAULT_NS_COEFFS), (12, (1.5, -0.5, 0.0))):
            got = newton_schulz_bf16(X, k, coeffs, rounding=lambda v: v)
            want = ref.newton_schulz(X, k, tuple(float(np.float32(c)) for c in coeffs))
            assert _rel(got, want) < 2e-5, (shape, k, _rel(got, want))


def test_bf16_error_is_that_of_bf16_operands():
    rng = np.random.default_rng(82)
    X = rng.standard_normal((96, 384)) * np.exp(0.5 * rng.standard_normal(384))[None, :]
    err = _rel(newton_schulz_bf16(X), ref.newton_schulz(X))
    assert 1e-3 < err < 1.5e-2, err
