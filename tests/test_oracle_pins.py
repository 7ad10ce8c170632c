"""The oracle against its pins (CPU only)."""
import pytest

import oracle
from tests.oracle_pins import ALL_PINS, BASIS_PINS


@pytest.mark.parametrize("pin", ALL_PINS, ids=lambda p: p.__name__)
def test_pin(pin):
    pin(oracle)


@pytest.mark.parametrize("pin", BASIS_PINS, ids=lambda p: p.__name__)
def test_basis_pin(pin):
    pin(oracle.basis_oracle)
