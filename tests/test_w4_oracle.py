"""The W4BF16 oracle against its pins (tests/w4_oracle_pins.py)."""
import pytest

from oracle import w4_oracle as W
from tests import w4_oracle_pins as P


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=[p.__name__ for p in P.ALL_PINS])
def test_pin(pin):
    pin(W)
