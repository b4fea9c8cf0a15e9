"""The fp64 oracle against its pins (hand-derived examples, library routines,
closed forms and invariants); see tests/oracle_pins.py for what each pins."""
import pytest

from oracle_pins import PINS


@pytest.mark.parametrize("name", list(PINS))
def test_oracle_pin(oracle_lib, name):
    PINS[name](oracle_lib)
