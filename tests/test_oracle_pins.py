"""The oracle against its pins (brute force, exact arithmetic, closed forms,
invariants and the paper's scan theorems).  CPU only."""
import pytest

import pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(pin):
    pin()
