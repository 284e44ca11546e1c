"""The fp64 oracle against facts fixed outside it (CPU only)."""
import pytest

from pins import PINS


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_oracle_pin(pin, oracle):
    pin(oracle)
