"""The score contract against the paper's definition of the score (Sec. 4.3, Eq. 3), on every
workload state the GPU parity tests compare: each contract score lies within SCORE_FP64_TOL of
the fp64 cosine, every kept-set difference between BottomK on contract scores and BottomK on
fp64 scores is a near-tie at the keep/evict boundary, and the number of such differences is the
one recorded in tests/golden/contract_vs_fp64.txt (written from the oracle by
tests/golden/make_contract_vs_fp64.py).  CPU only."""
import os

import pytest

import contract_fp64 as C

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "contract_vs_fp64.txt")


def _recorded():
    rows = {}
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        name, scored, _max_abs, diff = line.split()
        rows[name] = (int(scored), int(diff))
    return rows


def test_recorded_cases_cover_every_state():
    assert set(_recorded()) == set(C.CASES)


@pytest.mark.parametrize("name", list(C.CASES))
def test_contract_scores_match_fp64_definition(name):
    r = C.CASES[name]()
    scored, diff = _recorded()[name]
    assert r["scored"] == scored > 0
    assert r["max_abs"] <= C.SCORE_FP64_TOL, r
    assert r["unexplained"] == 0, r
    assert r["disagree"] == diff, r
