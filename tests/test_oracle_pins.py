"""The fp64 oracle against what the definition and mathematics fix (CPU only)."""
import pytest

import oracle
from tests import oracle_pins as P


@pytest.fixture(scope="module")
def orc():
    return oracle.default()


@pytest.mark.parametrize("check", P.ALL_CHECKS, ids=lambda c: c.__name__)
def test_oracle_pin(orc, check):
    check(orc)
