"""The CPU oracle against its pins (brute force, torch fp64, closed forms,
invariants, hand-worked examples). No GPU."""
import pytest

import oracle_pins as P


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin()
