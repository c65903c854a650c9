"""The oracle against its pins (CPU only): brute force, library routines, the
paper's counts and worked example.  See ``oracle_pins.py`` for what each pins."""
import pytest

import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)
