"""Failure detection without a fault: every device wait in the library is
bounded, and an expired wait is reported to the host as MALIB_ETIMEOUT by the
next sync while the context stays usable. The self-test waits on an mbarrier
phase that nothing completes, with a limit of a few milliseconds, so the wait
ends by its own limit; nothing traps, faults or hangs."""
import numpy as np
import pytest

import workloads
from gpu_util import context, load_population, need_gpu

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MalibError


def test_expired_wait_is_reported_and_context_survives():
    need_gpu()
    w = workloads.kuhn(n_episodes=2000)
    ctx = context()
    load_population(ctx, w)
    before = ctx.eval_payoff(w.pair_ids, w.n_episodes, w.seed)
    ctx.selftest_wait(False, 2_000_000)
    with pytest.raises(MalibError, match="ETIMEOUT"):
        ctx.sync()
    ctx.sync()                                   # the flag was cleared when it was read
    after = ctx.eval_payoff(w.pair_ids, w.n_episodes, w.seed)
    np.testing.assert_array_equal(after, before)
    ctx.close()


def test_completed_wait_reports_nothing():
    need_gpu()
    ctx = context()
    for _ in range(3):
        ctx.selftest_wait(True, 1_000_000)
    ctx.sync()
    ctx.close()


@pytest.mark.parametrize("limit", [0, -5, 1_000_000_001])
def test_wait_limit_is_checked_on_the_host(limit):
    need_gpu()
    ctx = context()
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.selftest_wait(False, limit)
    ctx.sync()
    ctx.close()
