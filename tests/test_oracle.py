"""The fp64 oracle against what the paper and mathematics fix (CPU only)."""
import numpy as np
import pytest

from oracle import rolekv_oracle as O
from tests import oracle_pins as P


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(pin):
    pin(O, np.random.default_rng(20260713))
