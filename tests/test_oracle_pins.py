"""The fp64 oracle against the paper's worked example, closed forms,
invariants, special cases and brute force on tiny inputs (CPU only)."""
import pytest

import oracle_pins as pins


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_oracle_pin(check):
    check()
