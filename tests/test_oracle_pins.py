"""The CPU oracle against its pins (closed forms, identities, brute force, invariants,
a hand-derived worked example, App. D storage figures, textbook attention)."""
import pytest

import oracle.densitykv as O
import oracle_pins as P


@pytest.mark.parametrize("check", P.ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(check):
    check(O)
