"""The float64 oracle against closed forms, invariants, library special cases,
finite differences and hand-worked examples (see oracle_pins.py)."""

import pytest

import oracle.grpo_objective as O
from oracle_pins import ALL_PINS


@pytest.mark.parametrize("pin", ALL_PINS, ids=[p.__name__ for p in ALL_PINS])
def test_pin(pin):
    pin(O)
