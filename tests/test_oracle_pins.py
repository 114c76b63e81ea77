"""The CPU oracle against the paper's fixed points, closed forms and brute force (no GPU)."""
import pytest

from tests import oracle_checks as C


@pytest.mark.parametrize("check", C.ALL_CHECKS, ids=lambda f: f.__name__)
def test_oracle_pin(check):
    check()
