"""The CPU oracle against its pins (no GPU)."""
import numpy as np
import pytest

import oracle
from oracle_pins import ALL_PINS


@pytest.fixture(scope="module")
def orc():
    return oracle.default()


@pytest.mark.parametrize("pin", ALL_PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)


def test_bad_arguments_rejected(orc):
    Q = np.zeros((4, 4), np.int8)
    s = np.ones(4, np.float32)
    with pytest.raises(ValueError):
        orc.project(Q, s, 4, 4, np.zeros(4, np.uint8), "nope")
    with pytest.raises(ValueError):
        orc.project(Q, s, 8, 4, np.zeros(4, np.uint8), "u8")   # Q too small
    with pytest.raises(ValueError):
        orc.project(Q, s, 4, 4, np.zeros(2, np.uint8), "u8")   # x too short
