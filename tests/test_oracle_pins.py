"""The float64 oracle against facts the paper and mathematics fix (CPU only)."""
import numpy as np
import pytest

import oracle
import pins


@pytest.fixture(scope="module")
def o():
    return oracle.default()


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda p: p.__name__)
def test_pin(o, pin):
    assert pin(o) == []


def test_rejects_invalid_arguments(o):
    x = np.zeros((1, 6))
    with pytest.raises(oracle.OracleError):
        o.fc_forward(x, np.zeros((1, 4, 6)), np.full((1, 3), 4, np.uint8))  # code >= K
    with pytest.raises(oracle.OracleError):
        o.conv_forward(np.zeros((1, 2, 2, 2)), np.zeros((1, 2, 2)),
                       np.zeros((1, 9, 1), np.uint8), 3, 3, 1, 0)  # kernel larger than map
    with pytest.raises(oracle.OracleError):
        o.fc_forward(x, np.zeros((2, 300, 3)), np.zeros((2, 3), np.uint8))  # K > 256
