"""The oracle against the hand-derived fixtures of tests/golden/."""
import pytest

from _golden import check, fixture_files, load


@pytest.mark.parametrize("path", fixture_files(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_oracle_matches_hand_derived_fixture(oracle_lib, path):
    case, expect = load(path)
    res = oracle_lib.validate(case["cand"], case["ref"], inputs=case["inputs"],
                              rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                              first_k=case["first_k"])
    check(res, expect)
