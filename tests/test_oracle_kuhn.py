"""Pins for the oracle's Kuhn poker: closed-form values of deterministic
profiles, Kuhn's (1950) equilibrium family worth -1/18 to the first player, a
brute-force enumeration written independently here, and Monte-Carlo agreement
with the exact value."""
import itertools

import numpy as np
import pytest

import workloads


def nash(alpha):
    # infoset index card*2 + h; J=0, Q=1, K=2; h=1 means facing a bet.
    p0 = np.array([alpha, 0.0, 0.0, alpha + 1 / 3, 3 * alpha, 1.0], np.float32)
    p1 = np.array([1 / 3, 0.0, 0.0, 1 / 3, 1.0, 1.0], np.float32)
    return p0, p1


@pytest.mark.parametrize("alpha", [0.0, 0.1, 0.25, 1 / 3])
def test_kuhn_nash_value(orc, alpha):
    p0, p1 = nash(alpha)
    assert abs(orc.kuhn_exact(p0, p1) - (-1 / 18)) < 1e-7


def test_kuhn_deterministic_profiles(orc):
    ones, zeros = np.ones(6, np.float32), np.zeros(6, np.float32)
    # both always bet/call: every hand is a showdown for 2; symmetric -> 0
    assert abs(orc.kuhn_exact(ones, ones) - 0.0) < 1e-12
    # nobody ever bets: showdown for 1 -> 0
    assert abs(orc.kuhn_exact(zeros, zeros) - 0.0) < 1e-12
    # seat 0 always bets, seat 1 never calls -> +1
    assert abs(orc.kuhn_exact(ones, zeros) - 1.0) < 1e-12
    # seat 0 passes and folds, seat 1 always bets -> -1
    assert abs(orc.kuhn_exact(zeros, ones) + 1.0) < 1e-12
    # seat 0 bets only with K (and calls with K), seat 1 calls only with K.
    p0 = np.array([0, 0, 0, 0, 1, 1], np.float32)
    p1 = np.array([0, 0, 0, 0, 1, 1], np.float32)
    # deals (c0,c1): (J,Q) pass,pass -> -1; (J,K) pass, bet(K), fold -> -1;
    # (Q,J) pass,pass -> +1; (Q,K) pass, bet, fold -> -1;
    # (K,J) bet, fold -> +1; (K,Q) bet, fold -> +1.   mean = 0/6
    assert abs(orc.kuhn_exact(p0, p1)) < 1e-12


def brute_force(p0, p1):
    """Independent enumeration over deals and every action sequence."""
    total = 0.0
    for c0, c1 in itertools.permutations(range(3), 2):
        sd = 1 if c0 > c1 else -1
        for seq in itertools.product([0, 1], repeat=3):
            prob, pay = 1.0 / 6, None
            a0 = seq[0]
            prob *= p0[c0 * 2] if a0 else 1 - p0[c0 * 2]
            a1 = seq[1]
            if a0:
                prob *= p1[c1 * 2 + 1] if a1 else 1 - p1[c1 * 2 + 1]
                pay = 2 * sd if a1 else 1
                if seq[2]:
                    continue
            else:
                prob *= p1[c1 * 2] if a1 else 1 - p1[c1 * 2]
                if not a1:
                    pay = sd
                    if seq[2]:
                        continue
                else:
                    a2 = seq[2]
                    prob *= p0[c0 * 2 + 1] if a2 else 1 - p0[c0 * 2 + 1]
                    pay = 2 * sd if a2 else -1
            total += prob * pay
    return total


def test_kuhn_exact_vs_brute_force(orc):
    rng = np.random.default_rng(1)
    for _ in range(50):
        p0 = rng.random(6, dtype=np.float32)
        p1 = rng.random(6, dtype=np.float32)
        assert abs(orc.kuhn_exact(p0, p1) - brute_force(p0.astype(float), p1.astype(float))) < 1e-12


def test_kuhn_mc_within_4se_of_exact(orc):
    w = workloads.kuhn()
    tables = np.stack([p.params for p in w.policies])
    res, _ = orc.kuhn_eval(tables, w.pair_ids, 10_000, w.seed)
    for k, (i, j) in enumerate(w.pair_ids):
        ex = orc.kuhn_exact(tables[i], tables[j])
        assert abs(res[k, 0] - ex) <= 4 * res[k, 1], (k, res[k], ex)
    # all n = 10,000 payoffs are integers in {-2,-1,1,2}: sums are integral
    assert np.all(res[:, 2] == np.round(res[:, 2]))
    assert np.all(np.abs(res[:, 0]) <= 2)


def test_kuhn_trace_consistency_and_deal_distribution(orc):
    """Each traced hand's payoff follows from its cards and actions, seats
    alternate, and the 6 deals are equally likely."""
    w = workloads.kuhn()
    tables = np.stack([p.params for p in w.policies])
    n = 6000
    res, tr = orc.kuhn_eval(tables, w.pair_ids[:1], n, 77, n_trace=n)
    tr = tr[0]
    outcome = {  # action sequence -> payoff in units of the showdown sign (None: fixed)
        (0, 0): ("sd", 1), (0, 1, 0): ("fix", -1), (0, 1, 1): ("sd", 2),
        (1, 0): ("fix", 1), (1, 1): ("sd", 2)}
    deals = np.zeros((3, 3), int)
    for row in tr:
        c0, c1, nd = row[0], row[1], row[2]
        acts = tuple(int(a) for a in row[3:3 + nd])
        kind, v = outcome[acts]
        want = v * (1 if c0 > c1 else -1) if kind == "sd" else v
        assert row[6] == want
        assert c0 != c1
        deals[c0, c1] += 1
    assert res[0, 2] == tr[:, 6].sum()
    cnt = deals[deals > 0]
    assert cnt.size == 6
    chi2 = ((cnt - n / 6) ** 2 / (n / 6)).sum()
    assert chi2 < 25.0      # 5 dof


def test_kuhn_entry_statistics(orc):
    """The payoff entry (mean, standard error, sum, sum of squares) equals the
    textbook estimators over the traced per-episode payoffs."""
    rng = np.random.default_rng(2)
    p0 = rng.random(6, dtype=np.float32)
    p1 = rng.random(6, dtype=np.float32)
    n = 2000
    res, tr = orc.kuhn_eval(np.stack([p0, p1]), np.array([[0, 1]]), n, 5, n_trace=n)
    r = tr[0, :, 6].astype(np.float64)
    assert res[0, 2] == r.sum()
    assert res[0, 3] == (r ** 2).sum()
    assert abs(res[0, 0] - r.mean()) < 1e-15
    assert abs(res[0, 1] - r.std(ddof=1) / np.sqrt(n)) < 1e-12


def test_kuhn_hands_at_any_id_match_the_evaluation(orc):
    """The per-id helper replays the evaluation's hands: pair k's hand e is the
    hand with global id k * n_episodes + e, and its payoffs sum to the entry's."""
    w = workloads.kuhn(n_episodes=500)
    tables = np.stack([p.params for p in w.policies])
    res, tr = orc.kuhn_eval(tables, w.pair_ids[:3], 500, 11, n_trace=500)
    for k in range(3):
        i, j = w.pair_ids[k]
        got = orc.kuhn_hands(tables[i], tables[j], k * 500, 500, 11)
        np.testing.assert_array_equal(got, tr[k])
        assert got[:, 6].sum() == res[k, 2]
    far = orc.kuhn_hands(tables[0], tables[1], (1 << 33) + 5, 64, 11)
    assert set(np.unique(far[:, 6])) <= {-2, -1, 1, 2}
    assert not np.array_equal(far, orc.kuhn_hands(tables[0], tables[1], 5, 64, 11))
