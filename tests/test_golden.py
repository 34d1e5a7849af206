"""CPU checks of the oracle against the fixtures of tests/golden: Kuhn's (1950)
equilibrium family and value (a published result, not the oracle's), and the
stored exact Leduc table (written by tests/golden/make_golden.py from the
oracle: a regression guard, so a change of the oracle's arithmetic shows here
and needs a new fixture with its justification)."""
import os
import sys

import numpy as np

import golden_data

sys.path.insert(0, os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden"))


def test_kuhn_equilibrium_family_value(orc):
    value, first, second = golden_data.kuhn_equilibrium()
    assert abs(value + 1 / 18) < 1e-15
    assert len(first) == 4 and second is not None
    for p0 in first:
        assert abs(orc.kuhn_exact(p0, second) - value) < 1e-7


def test_leduc_exact_table_reproduces(orc):
    import make_golden
    w = make_golden.leduc_population()
    params = [p.params for p in w.policies]
    rows = golden_data.leduc_exact_small()
    assert [(i, j) for i, j, _ in rows] == [tuple(int(x) for x in p) for p in w.pair_ids]
    for i, j, v in rows:
        assert abs(orc.leduc_exact(params[i], params[j], w.policies[0].dims) - v) < 1e-12
    # seat-0 payoffs lie within the game's range (a fold costs at least 1, the pot is at most 13)
    assert all(-13 <= v <= 13 for _, _, v in rows)
