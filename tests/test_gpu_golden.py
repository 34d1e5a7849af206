"""GPU evaluation against the fixtures of tests/golden, without running the
oracle: the Kuhn equilibrium family's value (exact-expectation mode within
1e-6, Monte Carlo within 4 standard errors) and the stored exact Leduc table
(Monte Carlo with 262,144 hands per pair within 4 standard errors)."""
import os
import sys

import numpy as np
import pytest

import golden_data
import workloads
from gpu_util import context, load_population, need_gpu

sys.path.insert(0, os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden"))

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_EXACT_EXPECTATION


def test_kuhn_equilibrium_family():
    need_gpu()
    value, first, second = golden_data.kuhn_equilibrium()
    w = workloads.Workload("kuhn_golden", workloads.ENV_KUHN, 2, 0, 0, 2, 0, 0)
    w.policies = [workloads.Policy(workloads.POL_TABULAR, workloads.F32, 0, (6, 0, 0, 1), p)
                  for p in first]
    w.policies.append(workloads.Policy(workloads.POL_TABULAR, workloads.F32, 1, (6, 0, 0, 1), second))
    ctx = context()
    load_population(ctx, w)
    pairs = np.array([[i, len(first)] for i in range(len(first))], np.int32)
    ex = ctx.eval_payoff_ex(pairs, 0, 0, MALIB_EXACT_EXPECTATION)
    assert np.abs(ex[:, 0] - value).max() < 1e-6
    mc = ctx.eval_payoff(pairs, 100_000, 17)
    assert np.all(np.abs(mc[:, 0] - value) < 4 * mc[:, 1])
    ctx.close()


def test_leduc_exact_table():
    need_gpu()
    import make_golden
    w = make_golden.leduc_population()
    rows = golden_data.leduc_exact_small()
    ctx = context()
    load_population(ctx, w)
    res = ctx.eval_payoff(w.pair_ids, 262_144, 23)
    for k, (_, _, v) in enumerate(rows):
        assert abs(res[k, 0] - v) < 4 * res[k, 1], (k, res[k], v)
        assert res[k, 1] < 0.01
    ctx.close()
