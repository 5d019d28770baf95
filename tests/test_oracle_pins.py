"""The oracle against closed forms, the paper's worked example, invariants
and brute force (no GPU)."""
import pytest

import oracle.memdecay_oracle as om
from tests import oracle_checks as oc


@pytest.mark.parametrize("check", oc.ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(check):
    check(om)
