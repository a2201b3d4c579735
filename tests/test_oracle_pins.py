"""The float64 oracle against facts the paper and mathematics fix (CPU only)."""
import pytest

import oracle.spade_oracle as O
from tests import oracle_pins as pins


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda f: f.__name__)
def test_oracle_pin(check):
    check(O)
