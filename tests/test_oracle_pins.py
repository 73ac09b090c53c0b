"""The fp64 oracle against closed forms, invariants, brute force, finite
differences and an independent PyTorch fp64 composition (CPU only)."""
import pytest

import oracle.solo_oracle as orc
from tests.oracle_pins import PINS


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin(orc)
