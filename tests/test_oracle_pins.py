"""The oracle against its pins (hand-worked values, brute force, closed
forms, invariants).  CPU only."""

import pytest

import pin_checks as P


@pytest.mark.parametrize("check", P.ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(oracle_mod, check):
    check(oracle_mod)
