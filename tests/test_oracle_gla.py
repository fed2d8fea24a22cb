"""The oracle's FEM read over a GLA prior against the paper's statements (CPU only)."""
import pytest

from tests import oracle_gla_pins


@pytest.mark.parametrize("check", oracle_gla_pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_gla_pin(check):
    check()
