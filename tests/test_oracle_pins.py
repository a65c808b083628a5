"""The fp64 oracle against what the paper and mathematics fix (CPU only)."""
import pytest

import oracle
from tests import oracle_pins


@pytest.fixture(scope="module")
def orc():
    return oracle.default()


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(orc, pin):
    pin(orc)


def test_oracle_rejects_bad_arguments(orc):
    import numpy as np
    q = np.zeros((0, 4))
    with pytest.raises(ValueError):
        orc.fwd(q, q, q, 0.5)
    x = np.zeros((3, 2))
    with pytest.raises(ValueError):
        orc.fwd(x, x, x, 0.5, tau_s=0.0)
    with pytest.raises(ValueError):
        orc.fwd_rows(x, x, x, [3], 0.5)
