"""The oracle agrees with every pin (closed forms, invariants, brute force, fixtures)."""
import pytest

from oracle import taskpress_oracle as O
from tests import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(O)
