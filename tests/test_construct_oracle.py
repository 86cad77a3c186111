"""Pins of the construction oracle (oracle/construct.py; paper Section 3.4,
Algorithm 1) against what the paper and the mathematics fix, CPU only.  The
checks themselves live in construct_pins.py, which lists them with their
sources; test_construct_mutants.py runs the same checks on planted mistakes
in copies of the oracle."""

import pytest

from oracle import construct as oc
from tests import construct_pins


@pytest.mark.parametrize("check", construct_pins.ALL_CHECKS, ids=lambda f: f.__name__[len("check_"):])
def test_construction_oracle_pin(check):
    check(oc)
