"""The fp64 oracle against its pins (library routines, closed forms, golden
values, brute force, invariants). CPU only."""
import pytest

import oracle_pins as pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(orc, pin):
    pin(orc)
