"""The oracle against what the paper and the mathematics fix (CPU only)."""
import pytest

import oracle_pins as P
from oracle import xshare_oracle as O


@pytest.mark.parametrize("check", P.ALL_CHECKS, ids=lambda c: c.__name__)
def test_pin(check):
    check(O)
