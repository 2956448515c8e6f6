"""The float64 oracle against what the paper and the mathematics fix (CPU)."""
import pytest

import pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda f: f.__name__[4:])
def test_pin(pin):
    pin()
