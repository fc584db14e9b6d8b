"""Pins of the counts-consumer oracle (MaxVio, App. E; REM replica allocation,
Sec. 3.2 Eq. benefit_score and App. B.1 Algorithm rem_allocation) against
examples worked by hand from the definitions, the paper's reading of a MaxVio
value, and invariants every allocation must keep."""
import json
import os

import numpy as np
import pytest

from oracle import rem

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def golden():
    return json.load(open(os.path.join(GOLDEN, "rem_worked_examples.json")))


def test_maxvio_ten_percent_reading():
    g = golden()["maxvio_ten_percent"]
    assert rem.maxvio(g["loads"]) == pytest.approx(g["maxvio"], abs=1e-15)


def test_maxvio_closed_forms():
    assert rem.maxvio([7, 7, 7, 7]) == 0.0                 # uniform
    assert rem.maxvio([0, 0, 0, 12]) == pytest.approx(3.0)  # one rank holds all: |R| - 1
    assert rem.maxvio([0, 10]) == pytest.approx(1.0)        # an idle rank counts as well
    assert rem.maxvio([0, 0, 0]) == 0.0                      # no tokens, no violation


def test_rank_loads_sum_the_resident_experts():
    counts = [5, 1, 7, 3, 9]
    assert rem.rank_loads(counts, [1, 0, 1, 2, 0], 3) == [10, 12, 3]


def test_benefit_score_cases():
    # case 1: receiver below tau, sender above: the smallest of the three gaps
    assert rem.benefit_score(T_e=100, L_s=90, L_r=10, tau=40) == 30
    assert rem.benefit_score(T_e=100, L_s=50, L_r=10, tau=40) == 10
    assert rem.benefit_score(T_e=7, L_s=90, L_r=10, tau=40) == 7
    # case 2: receiver at or above tau, sender above the receiver: half the gap, floored
    assert rem.benefit_score(T_e=100, L_s=45, L_r=40, tau=40) == 2
    assert rem.benefit_score(T_e=1, L_s=60, L_r=41, tau=40) == 1
    # otherwise -1
    assert rem.benefit_score(T_e=100, L_s=30, L_r=10, tau=40) == -1
    assert rem.benefit_score(T_e=100, L_s=40, L_r=40, tau=40) == -1


@pytest.mark.parametrize("i", [0, 1])
def test_rem_allocation_worked_examples(i):
    ex = golden()["examples"][i]
    A, L = rem.rem_allocate(ex["loads"], ex["expert_tokens"], ex["expert_rank"], ex["D"])
    assert [list(a) for a in A] == ex["placements"]
    assert L == ex["loads_after"]
    assert rem.maxvio(ex["loads"]) == pytest.approx(ex["maxvio_before"], abs=1e-15)
    assert rem.maxvio(L) == pytest.approx(ex["maxvio_after"], abs=1e-15)


@pytest.mark.parametrize("seed", range(8))
def test_rem_allocation_invariants(seed):
    rng = np.random.default_rng(seed)
    R, E, D = int(rng.integers(2, 9)), int(rng.integers(4, 40)), int(rng.integers(1, 4))
    home = rng.integers(0, R, E)
    tokens = rng.gamma(0.7, 500.0, E).round()
    loads = rem.rank_loads(tokens, home, R)
    A, L = rem.rem_allocate(loads, tokens, home, D)
    assert sum(L) == pytest.approx(sum(loads))              # tokens move, none appear
    per_rank = [0] * R
    moved = np.zeros(E)
    tau = sum(loads) / R
    for e, rs, rr, d in A:
        assert d > 0 and rs == home[e] and rr != rs
        per_rank[rr] += 1
        moved[e] += d
    assert max(per_rank) <= D
    assert (moved <= tokens + 1e-9).all()                   # never more than an expert holds
    assert len({(e, rr) for e, _, rr, _ in A}) == len(A)     # one replica of e per rank
    # every placement moves load from above the mean (or above the receiver) to
    # a receiver below it, so the busiest rank never gets busier
    assert max(L) <= max(loads) + 1e-9
    assert rem.maxvio(L) <= rem.maxvio(loads) + 1e-12
    assert tau == pytest.approx(sum(L) / R)
