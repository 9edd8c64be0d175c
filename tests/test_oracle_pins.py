"""The CPU oracle against the facts that pin it (runs without a GPU)."""
import pytest

import oracle.dsm_oracle as O
from oracle_pins import PINS


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin(O)


def test_worked_example_fp64_twin():
    import numpy as np
    from oracle_pins import pin_worked_example
    pin_worked_example(O, dt=np.float64)
