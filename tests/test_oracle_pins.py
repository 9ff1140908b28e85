"""The fp64 oracle against hand-derived examples, library routines, closed
forms and invariants of Section 3.1 / Eq. 1 (CPU only)."""
import pytest

import oracle_pins
from oracle import load


@pytest.fixture(scope="module")
def orc():
    return load()


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)
