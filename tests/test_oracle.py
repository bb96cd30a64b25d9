"""The CPU oracle against its pins (closed forms, library routines, the
paper's printed budgets, invariants and brute force).  No GPU needed."""
import pytest

from oracle_pins import ALL_PINS


@pytest.mark.parametrize("pin", ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin()
