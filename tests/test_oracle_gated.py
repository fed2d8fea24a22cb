"""The oracle's two-level gated read against the paper's statements (CPU only)."""
import pytest

import oracle
from tests import oracle_gated_pins


@pytest.fixture(scope="module")
def lib():
    return oracle.load()


@pytest.mark.parametrize("check", oracle_gated_pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_gated_pin(lib, check):
    check(lib)
