"""Pins for the oracle's Leduc hold'em: hand-worked hands, the exhaustive
betting tree (49 terminal action sequences, legal masks, chip bounds), exact
expectations of deterministic profiles worked by hand, and Monte-Carlo agreement
with the exact tree expectation."""
import itertools

import numpy as np
import pytest

import workloads

F, C, R = 0, 1, 2
J0, J1, Q0, Q1, K0, K1 = range(6)


@pytest.mark.parametrize("cards,actions,payoff0,contrib,ndec", [
    # J vs K, public Q, all checks: K high wins 1
    ((J0, K0, Q0), [C, C, C, C], -1, (1, 1), 4),
    # raise/call both rounds: 1+2 then +4 = 7 each, K wins
    ((J0, K0, Q0), [R, C, R, C], -7, (7, 7), 4),
    # J pairs the public J after the maximum pot: 13 each
    ((J0, K0, J1), [R, R, C, C, R, R, C], 13, (13, 13), 7),
    # eight decisions: check-raise-reraise-call in both rounds
    ((Q0, J0, K0), [C, R, R, C, C, R, R, C], 13, (13, 13), 8),
    # seat 1 folds to the opening raise: seat 0 wins seat 1's ante
    ((J0, K0, Q0), [R, F], 1, (3, 1), 2),
    # seat 0 folds facing a bet after checking
    ((K0, J0, Q0), [C, R, F], -1, (1, 3), 3),
    # round 2: check, raise to 5, re-raise to 9, fold: seat 0 gains seat 1's 5
    ((J0, Q0, K0), [C, C, C, R, R, F], 5, (9, 5), 6),
    # equal private ranks, no pair: split
    ((Q0, Q1, K0), [C, C, R, C], 0, (5, 5), 4),
    # seat 1 pairs the public card and wins over a higher private rank
    ((K0, J0, J1), [C, C, C, C], -1, (1, 1), 4),
])
def test_leduc_hand_worked(orc, cards, actions, payoff0, contrib, ndec):
    r = orc.leduc_play(*cards, actions)
    assert r["used"] == ndec == len(actions)
    assert r["done"]
    assert r["payoff0"] == payoff0
    assert r["contrib"] == contrib


def test_leduc_illegal_actions(orc):
    assert orc.leduc_play(J0, K0, Q0, [F])["used"] == -1           # no bet to fold to
    assert orc.leduc_play(J0, K0, Q0, [R, R, R])["used"] == -1     # third raise
    assert orc.leduc_play(J0, K0, Q0, [C, R, R, R])["used"] == -1
    r = orc.leduc_play(J0, K0, Q0, [R, R, C, R, R])
    assert r["used"] == 5 and not r["done"]


def test_leduc_observations(orc):
    r = orc.leduc_play(J0, K0, Q1, [C, R, C, R])
    o = r["obs"]
    # seat 0, J, round 1, no public card, 1 / 1, no raises, legal call+raise
    np.testing.assert_array_equal(o[0], np.float32([1, 0, 0, 0, 0, 0, 1, 1, 0, 1 / 13, 1 / 13,
                                                    1, 0, 0, 0, 1, 1]))
    # seat 1, K, facing nothing yet (check), may raise
    np.testing.assert_array_equal(o[1], np.float32([0, 0, 1, 0, 0, 0, 1, 1, 0, 1 / 13, 1 / 13,
                                                    1, 0, 0, 0, 1, 1]))
    # seat 0 facing the raise: own 1, opp 3, one raise, fold legal
    np.testing.assert_array_equal(o[2], np.float32([1, 0, 0, 0, 0, 0, 1, 1, 0, 1 / 13, 3 / 13,
                                                    0, 1, 0, 1, 1, 1]))
    # round 2, seat 0 first, public Q visible, 3 / 3
    np.testing.assert_array_equal(o[3], np.float32([1, 0, 0, 0, 1, 0, 0, 0, 1, 3 / 13, 3 / 13,
                                                    1, 0, 0, 0, 1, 1]))
    assert list(r["seats"]) == [0, 1, 0, 0]


def walk(orc, prefix, out):
    """All legal action sequences from the start (cards fixed: J vs K, Q)."""
    for a in (F, C, R):
        seq = prefix + [a]
        r = orc.leduc_play(J0, K0, Q0, seq)
        if r["used"] == -1:
            continue
        if r["done"]:
            out.append((seq, r))
        else:
            walk(orc, seq, out)


def test_leduc_exhaustive_tree(orc):
    term = []
    walk(orc, [], term)
    # per round 9 terminal sequences (cc crc crrc crf crrf rc rrc rf rrf), 5 of
    # which go on: 4 round-1 folds + 5 * 9 = 49.
    assert len(term) == 49
    assert len({tuple(s) for s, _ in term}) == 49
    for seq, r in term:
        assert 2 <= len(seq) <= 8
        assert max(r["contrib"]) <= 13 and min(r["contrib"]) >= 1
        if seq[-1] != F:
            assert r["contrib"][0] == r["contrib"][1]
            assert abs(r["payoff0"]) == r["contrib"][0]
        else:
            loser = r["seats"][-1]
            assert r["payoff0"] == (-r["contrib"][0] if loser == 0 else r["contrib"][1])
        # legal masks: fold iff facing a bet, call always, raise iff < 2 raises
        for t in range(len(seq)):
            o, lg = r["obs"][t], r["legal"][t]
            own, opp = o[9] * 13, o[10] * 13
            assert lg[0] == (opp > own + 0.5) and lg[1] == 1
            assert lg[2] == (o[13] == 0)
            np.testing.assert_array_equal(o[14:17], lg.astype(np.float32))
            assert o[:3].sum() == 1 and o[3:7].sum() == 1 and o[7:9].sum() == 1
            assert o[11:14].sum() == 1


def test_leduc_deal_distribution(orc):
    seen = np.zeros((6, 6, 6), int)
    n = 24000
    for g in range(n):
        c0, c1, p = orc.leduc_deal(g, 4242)
        assert len({c0, c1, p}) == 3
        seen[c0, c1, p] += 1
    cnt = seen[seen > 0]
    assert cnt.size == 120
    chi2 = ((cnt - n / 120) ** 2 / (n / 120)).sum()
    assert chi2 < 190.0     # 119 dof, p ~ 1e-4


def const_policy(logits, dims=(17, 4, 4, 3)):
    """MLP whose logits are its last bias whatever the input."""
    i, h1, h2, o = dims
    p = np.zeros(workloads.mlp_param_count(dims), np.float32)
    p[-o:] = logits
    return p


def test_leduc_exact_deterministic_profiles(orc):
    dims = (17, 4, 4, 3)
    call = const_policy([-100, 100, -100])
    raise_ = const_policy([-100, 0, 100])       # raise when legal, else call
    fold = const_policy([100, 0, -100])         # fold facing a bet, else check
    # identical strategies regardless of cards: symmetric showdowns -> 0
    assert abs(orc.leduc_exact(call, call, dims)) < 1e-12
    assert abs(orc.leduc_exact(raise_, raise_, dims)) < 1e-12
    # seat 0 opens with a raise, seat 1 folds to it: +1 every hand
    assert abs(orc.leduc_exact(raise_, fold, dims) - 1.0) < 1e-12
    # seat 0 checks then folds to the raise: -1 every hand
    assert abs(orc.leduc_exact(fold, raise_, dims) + 1.0) < 1e-12


def test_leduc_exact_card_aware_profile(orc):
    """Seat 0 raises (when legal) only holding a K, else checks/calls; seat 1
    always checks/calls. Every hand then goes to showdown with pot 1, 3, 5 or
    7 ... computed here by a direct enumeration over the 120 deals."""
    dims = (17, 3, 3, 3)
    p = np.zeros(workloads.mlp_param_count(dims), np.float32)
    i, h1, h2, o = dims
    W1 = np.zeros((h1, i), np.float32); W1[0, 2] = 1.0          # h1[0] = [private K]
    W2 = np.eye(3, dtype=np.float32)
    W3 = np.zeros((o, h2), np.float32); W3[2, 0] = 200.0        # raise logit
    b3 = np.float32([-100, 0, -100])
    p[:] = np.concatenate([W1.ravel(), np.zeros(3), W2.ravel(), np.zeros(3), W3.ravel(), b3])
    call = const_policy([-100, 100, -100], dims)
    total = 0.0
    for c0, c1, pub in itertools.permutations(range(6), 3):
        r0, r1, rp = c0 // 2, c1 // 2, pub // 2
        pot = 7 if r0 == 2 else 1      # K: raise + call in each round -> 1+2+4
        if r0 == rp:
            w = 1
        elif r1 == rp:
            w = -1
        else:
            w = (r0 > r1) - (r0 < r1)
        total += w * pot / 120
    assert abs(orc.leduc_exact(p, call, dims) - total) < 1e-12


def test_leduc_mc_within_4se_of_exact(orc):
    w = workloads.leduc(pop=2, with_bias=True, seed=7)
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    res, _ = orc.leduc_eval(params, dims, w.pair_ids, 20_000, 99)
    for k, (i, j) in enumerate(w.pair_ids):
        ex = orc.leduc_exact(params[i], params[j], dims)
        assert abs(res[k, 0] - ex) <= 4 * res[k, 1], (k, res[k], ex)


def test_leduc_records_and_replay(orc):
    """Recorded hands are legal and consistent; replaying the oracle's own
    logits reproduces every action and payoff."""
    w = workloads.leduc(pop=2, seed=8)
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    res, rec = orc.leduc_eval(params, dims, w.pair_ids, 300, 5, n_rec=300)
    assert np.all((rec["ndec"] >= 2) & (rec["ndec"] <= 8))
    np.testing.assert_array_equal(res[:, 2], rec["payoff"].sum(1))
    res2, rec2 = orc.leduc_eval(params, dims, w.pair_ids, 300, 5, n_rec=300,
                                ext_logits=rec["logits"])
    np.testing.assert_array_equal(rec2["action"], rec["action"])
    np.testing.assert_array_equal(res2, res)
    # a replay with perturbed logits changes some actions (the draw uses them)
    res3, rec3 = orc.leduc_eval(params, dims, w.pair_ids, 300, 5, n_rec=300,
                                ext_logits=rec["logits"] * -1.0)
    assert np.any(rec3["action"] != rec["action"])
    for p in range(w.n_pairs):
        for e in range(50):
            nd = rec["ndec"][p, e]
            g = p * 300 + e
            cards = orc.leduc_deal(g, 5)
            r = orc.leduc_play(*cards, list(rec["action"][p, e, :nd]))
            assert r["used"] == nd and r["done"] and r["payoff0"] == rec["payoff"][p, e]
            np.testing.assert_array_equal(r["obs"], rec["obs"][p, e, :nd])
            np.testing.assert_array_equal(r["seats"], rec["seat"][p, e, :nd])
            lg = orc.mlp_forward(params[w.pair_ids[p][0]], dims, rec["obs"][p, e, :nd])
            mine = rec["seat"][p, e, :nd] == 0
            np.testing.assert_array_equal(lg[mine], rec["logits"][p, e, :nd][mine])
