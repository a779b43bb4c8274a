"""The oracle against its pins (closed forms, invariants, the paper's worked
example, Monte Carlo of the speculative-decoding rule).  CPU only."""
import pytest

import oracle
from oracle_pins import ALL_CHECKS


@pytest.fixture(scope="module")
def orc():
    return oracle.get()


@pytest.mark.parametrize("check", ALL_CHECKS, ids=lambda c: c.__name__[6:])
def test_pin(orc, check):
    check(orc)
