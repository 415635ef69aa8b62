"""The fp8 chunk oracle against facts that do not come from itself (no GPU)."""
import pytest

import oracle_pins_fp8 as pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(oracle_lib, pin):
    pin(oracle_lib)
