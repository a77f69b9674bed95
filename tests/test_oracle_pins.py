"""The oracle against what mathematics fixes (no GPU)."""
import pytest

import oracle
import oracle_pin_checks as pins


@pytest.fixture(scope="module")
def lib():
    return oracle.load()


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(lib, check):
    check(lib)
