"""Pins of the RL-stage reward shaping and advantages (Sec. 3.4): a case worked
by hand from the equations, and the invariants the paper states."""
import math

import numpy as np
import pytest

from oracle import cospec_rl as RL

P = RL.RLParams(alpha=1.0, beta=0.25, eta_fail=0.5, eps=1e-6)


def _hand_case():
    """One prompt, two rollouts, K = 3 (see the expected values below).
    Rollout 0 (correct), round 0: Delta = 1,0,0, a = 1,1,0 -> s = 3, i* = 2,
      rho = (3-2)/(4-2) = 1/2, I = {2, 3}, g = 1/2 each; round 1: no mismatch.
    Rollout 1 (incorrect), round 2: Delta = 0,1,0, a = 1,1,1 -> s = 4, I = {1, 3},
      both accepted: g = -|ell| = -2, -0.5; round 3: Delta = 0,0,1, a = 0,1,1 ->
      s = 1, I = {1}, the rejection: g = -0.25."""
    group_off = [0, 2]
    correct = [1, 0]
    round_off = [0, 2, 4]
    match = [[1, 0, 0], [1, 1, 1], [0, 1, 0], [0, 0, 1]]
    accept = [[1, 1, 0], [1, 1, 1], [1, 1, 1], [0, 1, 1]]
    ell = [[0.0, -1.0, -3.0], [0.0, 0.0, 0.0], [-2.0, 0.0, -0.5], [-1.5, -0.7, 0.0]]
    return group_off, correct, round_off, 3, match, accept, ell


def test_hand_worked_case():
    out = RL.rl_advantages(*_hand_case(), P)
    np.testing.assert_allclose(out["g"], [[0, 0.5, 0.5], [0, 0, 0], [-2.0, 0, -0.5], [-0.25, 0, 0]])
    assert out["rho"][0] == 0.5 and math.isnan(out["rho"][1])
    assert out["rho"][2] == 1.0 and out["rho"][3] == 0.0
    np.testing.assert_allclose(out["J"], [1.0, -2.75])
    # mixed group: gamma = 2.75 / 1.0 -> Jbar = (2.75, -2.75), mu = 0, sigma = 2.75
    np.testing.assert_allclose(out["Jbar"], [2.75, -2.75], rtol=1e-5)
    np.testing.assert_allclose(out["adv"], [1.0, -1.0], rtol=1e-5)
    np.testing.assert_allclose(out["adv_dec"], [[0, 0.5, 0.5], [0, 0, 0],
                                                [-2 / 2.75, 0, -0.5 / 2.75], [-0.25 / 2.75, 0, 0]],
                               rtol=1e-5)


def test_round_quantities_extremes():
    # whole block kept: s = K+1, rho = 1; first mismatch rejected: rho = 0
    s, i_star, i_rej, rho, eff = RL.round_quantities([1, 0, 1, 0], [1, 1, 1, 1], 4)
    assert (s, i_star, i_rej, rho, eff) == (5, 2, 5, 1.0, [2, 4])
    s, i_star, i_rej, rho, eff = RL.round_quantities([1, 0, 0, 0], [1, 0, 1, 0], 4)
    assert (s, i_star, i_rej, rho, eff) == (2, 2, 2, 0.0, [2])
    # no mismatch: nothing is effective
    assert RL.round_quantities([1, 1], [1, 1], 2)[3:] == (None, [])


def _random_batch(rng, groups, K, mode):
    group_off = [0]; correct = []; round_off = [0]
    match, accept, ell = [], [], []
    for x in range(groups):
        M = int(rng.integers(1, 6))
        for m in range(M):
            c = {"mixed": rng.random() < 0.5, "pos": True, "neg": False}[mode]
            correct.append(int(c))
            for r in range(int(rng.integers(1, 8))):
                d = (rng.random(K) < 0.6).astype(int)
                a = np.where(d == 1, 1, (rng.random(K) < 0.5).astype(int))
                match.append(list(d)); accept.append(list(a))
                ell.append(list(-rng.exponential(1.5, K)))
            round_off.append(len(match))
        group_off.append(len(correct))
    return group_off, correct, round_off, K, match, accept, ell


@pytest.mark.parametrize("mode", ["mixed", "pos", "neg"])
def test_group_invariants(mode):
    rng = np.random.default_rng({"mixed": 1, "pos": 2, "neg": 3}[mode])
    batch = _random_batch(rng, 40, 6, mode)
    out = RL.rl_advantages(*batch, P)
    group_off, correct = batch[0], batch[1]
    for x in range(len(group_off) - 1):
        ms = list(range(group_off[x], group_off[x + 1]))
        c = [correct[m] for m in ms]
        adv = out["adv"][ms]
        if len(ms) > 1:
            # standardised within the group: zero mean
            assert abs(adv.mean()) < 1e-6
        if 0 < sum(c) < len(c) and sum(out["J"][m] for m in ms if correct[m]) > 1e-3:
            # mixed (with some positive return to rebalance): the rebalanced
            # returns sum to 0 and keep their signs
            jb = out["Jbar"][ms]
            assert abs(jb.sum()) < 1e-4 * max(1.0, np.abs(jb).max())
            assert all((jb[i] >= 0) == bool(c[i]) or out["J"][ms][i] == 0 for i in range(len(ms)))
        if sum(c) == 0 and len(ms) > 1:
            # all incorrect: scaled by eta_fail against the plain standardisation
            j = out["J"][ms]
            sd = j.std()
            if sd > 1e-3:
                np.testing.assert_allclose(adv, 0.5 * (j - j.mean()) / (sd + 1e-6), rtol=1e-9)
    # decision advantages: correct rollouts rho * Adv, incorrect ones shares of Adv summing to Adv
    round_off = batch[2]
    for m in range(len(correct)):
        rs = range(round_off[m], round_off[m + 1])
        tot = sum(out["adv_dec"][r].sum() for r in rs)
        if not correct[m] and sum(np.abs(out["g"][r]).sum() for r in rs) > 0:
            assert abs(tot - out["adv"][m]) < 1e-9 * max(1.0, abs(out["adv"][m]))
        if correct[m]:
            for r in rs:
                for i in range(batch[3]):
                    if out["eff"][r, i]:
                        assert out["adv_dec"][r, i] == pytest.approx(out["rho"][r] * out["adv"][m])
    # effective decisions are exactly the mismatches up to the first rejection
    for r in range(len(batch[4])):
        s = RL.round_quantities(batch[4][r], batch[5][r], batch[3])[0]
        for i in range(1, batch[3] + 1):
            assert out["eff"][r, i - 1] == (batch[4][r][i - 1] == 0 and i <= min(s, batch[3]))


def test_objective_terms():
    batch = _hand_case()
    Rt, K = 4, 3
    ones = np.ones((Rt, K))
    out = RL.rl_advantages(*batch, P, ratio=ones, p_new=0.5 * ones, p_ref=0.5 * ones)
    surr, ent, kl, loss = out["loss_terms"]
    eff = out["eff"].astype(bool)
    # ratio 1: the surrogate is the sum of the decision advantages
    assert surr == pytest.approx(out["adv_dec"][eff].sum())
    # p = 1/2 everywhere: entropy log 2 per decision, KL 0
    assert ent == pytest.approx(eff.sum() * math.log(2))
    assert kl == 0.0
    assert loss == pytest.approx(-surr - 0.01 * ent)
    # clipping: a ratio of 2 on a positive advantage counts as 1 + 0.2
    r2 = ones.copy(); r2[0, 1] = 2.0
    out2 = RL.rl_advantages(*batch, P, ratio=r2, p_new=0.5 * ones, p_ref=0.5 * ones)
    assert out2["loss_terms"][0] == pytest.approx(surr + 0.2 * out["adv_dec"][0, 1])
    # KL of Bernoulli(0.9) against Bernoulli(0.5)
    assert RL.bernoulli_kl(0.9, 0.5) == pytest.approx(0.9 * math.log(1.8) + 0.1 * math.log(0.2))
