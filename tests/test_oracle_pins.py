"""The fp64 oracle against closed forms, special cases, golden files and a
library routine (no GPU)."""
import pytest

import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda p: p.__name__)
def test_pin_holds(oracle_mod, pin):
    assert pin(oracle_mod) == []
