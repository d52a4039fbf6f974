"""The fp64 oracle against its pins (CPU only)."""
import pytest

import oracle_pins as P


@pytest.mark.parametrize("pin", P.ALL_PINS + P.BRUTE_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(pin):
    pin()
