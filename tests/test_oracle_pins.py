"""The oracle against what the paper and the mathematics fix (CPU only)."""
import pytest

import oracle.malt_ref as ref
from tests import oracle_pins


@pytest.mark.parametrize("check", oracle_pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_oracle_pin(check):
    check(ref)
