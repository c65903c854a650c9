"""The oracle against its pins (CPU only): brute force, library routines, the
paper's counts and worked example.  See ``oracle_pins.py`` for what each pins."""
import pytest

import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)


def test_epilogue_by_hand():
    """oracle.epilogue: bias per output channel, then max(., 0); the error scale
    grows by |bias| (values worked by hand)."""
    import numpy as np
    import oracle
    Y = np.array([[1.0, -2.0, 0.25], [-3.0, 4.0, -0.25]])
    S = np.array([[1.0, 2.0, 3.0], [4.0, 5.0, 6.0]])
    Yr, Sr = oracle.epilogue(Y, S, bias=np.array([0.5, 1.0, -1.0]), relu=True)
    assert (Yr == np.array([[1.5, 0.0, 0.0], [0.0, 5.0, 0.0]])).all()
    assert (Sr == np.array([[1.5, 3.0, 4.0], [4.5, 6.0, 7.0]])).all()
    Yn, Sn = oracle.epilogue(Y, S)
    assert (Yn == Y).all() and (Sn == S).all()
    Yb, _ = oracle.epilogue(Y, S, bias=np.array([0.5, 1.0, -1.0]))
    assert (Yb == np.array([[1.5, -1.0, -0.75], [-2.5, 5.0, -1.25]])).all()
