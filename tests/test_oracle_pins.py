"""The fp64 oracle against facts fixed outside it (see oracle_pins.py)."""

import pytest

import oracle
from tests import oracle_pins


@pytest.mark.parametrize("check", oracle_pins.ALL_CHECKS, ids=lambda f: f.__name__)
def test_oracle_pin(check):
    oracle.use_library(None)
    check(oracle)
