"""The CPU oracle against its pins (no GPU needed)."""
import pytest

from oracle import rowop_oracle as orc
from tests.oracle_pins import ALL_PINS


@pytest.mark.parametrize("pin", ALL_PINS, ids=lambda p: p.__name__)
def test_oracle_pin(pin):
    pin(orc)


def test_oracle_rejects_bad_offsets():
    import numpy as np
    with pytest.raises(ValueError):
        orc.softmax_ragged(np.zeros(4), np.array([0, 3, 2, 4]))
    with pytest.raises(ValueError):
        orc.softmax_ragged(np.zeros(4), np.array([1, 4]))
    with pytest.raises(ValueError):
        orc.softmax_ragged(np.zeros(4), np.array([0, 5]))
